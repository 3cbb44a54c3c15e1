// Causal append-chunk attention on the 5th-generation tensor cores
// (tcgen05 + TMEM), for rows that append a tool-observation chunk (L > 1).
//
// One CTA per SM, persistent, 11 warps. A work item is 256 query rows of one
// append row and kv head: (256 / g) consecutive tokens x the g query heads of
// that kv head, held as two 128-row tiles A and B (TMEM lanes = rows). Both
// tiles read the same K/V stream, so each K/V block in shared memory feeds
// four MMA chains (S_A, S_B, O_A, O_B), and the K/V bytes per flop are half
// those of a one-tile CTA.
//   warps 0-3  softmax of tile A, warps 4-7 softmax of tile B: thread t owns
//              row t & 127 of its tile. Per 128-key block it reads the 128
//              scores from TMEM in two chunks of 64, keeps the running max and
//              row sum, writes P (bf16) to the tile's TMEM P buffer, and
//              rescales O (lazily: only when the max grows by more than 2^8;
//              a rise inside the second chunk rescales the first chunk's P in
//              place). The S buffer is released as soon as both chunks are in
//              registers. Epilogue: O / l and the log-sum-exp to global memory
//              (out in host memory, append_tc_kernel<*, true>: each row as
//              four 32-byte stores, whole sectors for the host link);
//   warp 8     TMA producer: item queue, both query tiles (one 3-D box of
//              (256 / g) tokens x g heads x 64 dims), and K and V blocks
//              (8 pages = 128 keys, 16 KiB) in two rings of their own: a K
//              block is released as soon as S_A and S_B have read it, a V block
//              only after both PVs, so K runs a block ahead of V and the
//              K/V loads are in flight for most of a ring's length (they
//              often wait on HBM, which takes microseconds under load);
//   warps 9, 10  MMA issuers of tile A and tile B: S_X(b) = Q_X K_b^T (M 128,
//              N 128, K 64, both operands K-major from shared memory), then
//              O_X += P_X(b - 1) V_(b-1) (M 128, N 64, K 128; P from TMEM,
//              V MN-major from shared memory).
// TMEM (512 columns): S_A, S_B (128 each), O_A, O_B, P_A, P_B (64 each).
//
// Ordering (all mbarriers, all waits bounded; X = tile A or B, phase = the
// CTA's running block count, so no waiter can fall two phases behind):
//   k_full/k_empty     K ring; a stage is released by the commits after S_A, S_B
//   v_full/v_empty     V ring; a stage is released by the commits after PV_A, PV_B
//   s_full[X]          S_X(b) complete (commit after its 4 MMAs)
//   s_free[X]          S_X(b) loaded into registers (4 warps arrive)
//   p_full[X]          P_X(b) stored and O_X rescaled (4 warps arrive)
//   o_ready[X]         PV_X(b) complete; also guards the single P buffer
//   o_free[X]          epilogue has read O_X (next item may overwrite it)
//   q_full/q_empty     query tiles loaded / last QK^T of the item done
//   item_full/empty[2] two-slot queue of work items from the producer
//
// A wait that runs out sets an abort flag in shared memory that every other
// role's waits poll, so the whole CTA leaves within microseconds; before TMEM
// is freed the issuers wait for their MMAs and the producer for its copies
// still in flight. append_tc_kernel<true, false> is the self-test form of the same
// kernel (mcpu_selftest_append_abort): one chosen role stops at the second
// key block of its first item and waits on a barrier nothing completes (for
// half the wait limit), and each warp reports when it left.
#include "tcgen05.cuh"

namespace mcpu {

constexpr int kTcRows = 128;                          // rows per tile (TMEM lanes)
constexpr int kTcKeys = 128;                          // keys per block
// Ring depths and the register cap leave room on every SM for one CTA of the
// memory-bound decode kernel (side stream): 145 KiB of shared memory here,
// and at most 3 warps x 144 registers on any SM sub-partition.
constexpr int kTcKStages = 4, kTcVStages = 3;
constexpr int kTcQBytes = kAppendTcRows * kRowBytes;  // both tiles: 32 KiB
constexpr int kTcTileQBytes = kTcRows * kRowBytes;    // 16 KiB
constexpr int kTcKvBytes = kTcKeys * kRowBytes;       // one K or V block: 16 KiB
constexpr int kTcProducerWarp = 8, kTcSWarp = 9, kTcPvWarp = 10;
constexpr int kTcThreads = 352;
constexpr uint32_t kTmemCols = 512;
// TMEM columns of tile x (0 = A, 1 = B)
__device__ __forceinline__ uint32_t col_s(int x) { return x ? 128u : 0u; }
__device__ __forceinline__ uint32_t col_o(int x) { return x ? 320u : 256u; }
__device__ __forceinline__ uint32_t col_p(int x) { return x ? 448u : 384u; }
constexpr float kRescaleThreshold = 8.f;  // log2 units: P may reach 2^8 before O is rescaled

static_assert(kAppendTcRows == 2 * kTcRows, "an item is two tiles");

struct TcSmem {  // barriers and small state, after the tiles
  uint64_t q_full, q_empty;
  uint64_t k_full[kTcKStages], k_empty[kTcKStages], v_full[kTcVStages], v_empty[kTcVStages];
  uint64_t s_full[2], s_free[2], p_full[2], o_ready[2], o_free[2];
  uint64_t item_full[2], item_empty[2];
  uint64_t drain[2];  // each issuer's last MMAs complete (before TMEM is freed)
  uint64_t never;     // self-test form only: a barrier nothing completes
  AppendItem items[2];
  int32_t item_idx[2];
  uint32_t tmem_base;
  int32_t abort_flag;  // 1: a wait ran out; 2: the self-test's stalled role gave up
  uint64_t t_start;    // self-test form only: %globaltimer at kernel start
};

size_t append_tc_smem_bytes() {
  return 1024 + kTcQBytes + (size_t)(kTcKStages + kTcVStages) * kTcKvBytes + sizeof(TcSmem);
}

namespace {

// Bounded wait that also gives up when another role has aborted. The polls
// sleep (the producer and the MMA issuers wait most of the time and share
// sub-partitions with the softmax warps). Used by the producer and issuers.
__device__ __forceinline__ bool wait_bar(uint32_t bar, uint32_t parity, volatile int32_t* abort_flag) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = global_timer_ns();
  while (!mbar_try_wait_sleep(bar, parity, 10000)) {
    if (*abort_flag) return false;
    if (global_timer_ns() - t0 > kWaitTimeoutNs) {
      *abort_flag = 1;
      return false;
    }
  }
  return true;
}

// The softmax warps' bounded wait: the same, with plain polls (no
// suspend-time hint). The softmax is the critical path and rarely waits
// long; a sleeping poll there made the mixed batch's step ~0.65 % slower.
__device__ __forceinline__ bool wait_bar_poll(uint32_t bar, uint32_t parity, volatile int32_t* abort_flag) {
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

// 64 scores of one chunk with a -inf mask where key j is not visible to the
// query at `pos` (window lower bound `lo`).
__device__ __forceinline__ void mask_chunk(uint32_t (&sv)[2][32], int kbase, int pos, int lo) {
#pragma unroll
  for (int c = 0; c < 2; ++c)
#pragma unroll
    for (int e = 0; e < 32; ++e) {
      const int j = kbase + 32 * c + e;
      if (j > pos || j < lo) sv[c][e] = 0xff800000u;
    }
}

__device__ __forceinline__ float chunk_max(const uint32_t (&sv)[2][32]) {
  float m[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
#pragma unroll
  for (int c = 0; c < 2; ++c)
#pragma unroll
    for (int e = 0; e < 32; e += 8)
#pragma unroll
      for (int k = 0; k < 4; ++k) m[k] = fmax3(m[k], __uint_as_float(sv[c][e + 2 * k]), __uint_as_float(sv[c][e + 2 * k + 1]));
  return fmaxf(fmaxf(m[0], m[1]), fmaxf(m[2], m[3]));
}

// p = 2^(s * scale_log2 - m) for the 64 scores, packed to bf16 pairs; returns
// the fp32 sum of the 64 values.
__device__ __forceinline__ float chunk_exp(const uint32_t (&sv)[2][32], float scale_log2, float neg_mu,
                                           uint32_t (&pk)[32]) {
  const uint64_t sl2x2 = pack_f32x2(scale_log2, scale_log2);
  const uint64_t nmux2 = pack_f32x2(neg_mu, neg_mu);
  uint64_t lsum[2] = {0, 0};
#pragma unroll
  for (int c = 0; c < 2; ++c)
#pragma unroll
    for (int e = 0; e < 32; e += 2) {
      const uint64_t x = fma2((uint64_t)sv[c][e] | ((uint64_t)sv[c][e + 1] << 32), sl2x2, nmux2);
      const float p0 = ex2_approx(lo_f32(x));
      const float p1 = ex2_approx(hi_f32(x));
      lsum[(e >> 1) & 1] = add2(lsum[(e >> 1) & 1], pack_f32x2(p0, p1));
      pk[c * 16 + e / 2] = pack_bf16x2(p0, p1);
    }
  const uint64_t ls = add2(lsum[0], lsum[1]);
  return lo_f32(ls) + hi_f32(ls);
}

__device__ __forceinline__ void st_shared_zero16(uint32_t addr) {
  asm volatile("st.shared.v4.u32 [%0], {%1, %1, %1, %1};" ::"r"(addr), "r"(0u) : "memory");
}
// one 32-byte store (p 32-byte aligned)
__device__ __forceinline__ void st_global_v8(void* p, const uint32_t* w) {
  asm volatile("st.global.v8.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8};" ::"l"(p), "r"(w[0]), "r"(w[1]), "r"(w[2]),
               "r"(w[3]), "r"(w[4]), "r"(w[5]), "r"(w[6]), "r"(w[7]) : "memory");
}

// Self-test form only: the stalled role waits on a barrier nothing completes
// for half the library's wait limit, without polling the abort flag; then it
// raises the flag with its own mark (2) unless another role already did. The
// other roles, which began waiting at about the same time with the full
// limit, must leave on seeing the flag; one that ran out of its own wait
// instead would overwrite the mark with 1, and leave a half limit later.
constexpr uint64_t kSelftestStallNs = kWaitTimeoutNs / 2;
__device__ __forceinline__ void selftest_stall(uint32_t never_bar, int32_t* abort_flag) {
  const uint64_t t0 = global_timer_ns();
  while (!mbar_try_wait_sleep(never_bar, 0, 10000)) {
    if (global_timer_ns() - t0 > kSelftestStallNs) break;
  }
  atomicCAS(abort_flag, 0, 2);
}

// Probabilities of one chunk against the running reference m_ref (log2
// units): p = 2^(s * scale_log2 - m_ref). The common path computes no max:
// a chunk sum below 2^8 proves every p is below 2^8, the bound the lazy
// rescale keeps. Otherwise (or before the first reference exists) the chunk
// max is taken; if it exceeds m_ref by more than the threshold, m_ref is
// raised, `alpha` is multiplied by the factor that rescales earlier
// probabilities, and the chunk is recomputed. Returns the chunk sum.
__device__ __forceinline__ float chunk_probs(const uint32_t (&sv)[2][32], float scale_log2, float& m_ref,
                                             float& alpha, uint32_t (&pk)[32]) {
  float lc = 0.f;
  bool redo = m_ref == -INFINITY;
  if (!redo) {
    lc = chunk_exp(sv, scale_log2, -m_ref, pk);
    redo = !(lc < 256.f);  // also for inf / NaN
  }
  if (redo) {
    const float mx = chunk_max(sv) * scale_log2;
    if (mx > m_ref + kRescaleThreshold) {  // also true for the first finite max
      alpha *= ex2_approx(m_ref - mx);     // 0 when m_ref == -inf
      m_ref = mx;
    }
    lc = chunk_exp(sv, scale_log2, m_ref == -INFINITY ? 0.f : -m_ref, pk);
  }
  return lc;
}

}  // namespace

// kOutHost: out lies in page-locked host memory (written over the host link)
template <bool kSelfTest, bool kOutHost>
__global__ void __maxnreg__(144)
    append_tc_kernel(const __grid_constant__ CUtensorMap kmap, const __grid_constant__ CUtensorMap vmap,
                     const __grid_constant__ CUtensorMap qmap, const AttnParams p) {
  // nothing to do (no append rows this call): leave before TMEM and barriers
  if (header(p)->n_append == 0) return;
  extern __shared__ uint8_t smem_raw[];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t raw = smem_addr(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  const uint32_t sQ = base;
  const uint32_t sK = base + kTcQBytes;
  const uint32_t sV = sK + kTcKStages * kTcKvBytes;
  TcSmem& st = *reinterpret_cast<TcSmem*>(smem_raw + (base - raw) + kTcQBytes +
                                          (kTcKStages + kTcVStages) * kTcKvBytes);
  volatile int32_t* abort_flag = &st.abort_flag;
  auto bar = [&](uint64_t& b) { return smem_addr(&b); };

  if (threadIdx.x == 0) {
    mbar_init(bar(st.q_full), 1);
    mbar_init(bar(st.q_empty), 2);  // one commit per tile issuer
    for (int s = 0; s < kTcKStages; ++s) {
      mbar_init(bar(st.k_full[s]), 1);
      mbar_init(bar(st.k_empty[s]), 2);
    }
    for (int s = 0; s < kTcVStages; ++s) {
      mbar_init(bar(st.v_full[s]), 1);
      mbar_init(bar(st.v_empty[s]), 2);
    }
    for (int x = 0; x < 2; ++x) {
      mbar_init(bar(st.s_full[x]), 1);
      mbar_init(bar(st.s_free[x]), 4);
      mbar_init(bar(st.p_full[x]), 4);
      mbar_init(bar(st.o_ready[x]), 1);
      mbar_init(bar(st.o_free[x]), 4);
      mbar_init(bar(st.item_full[x]), 1);
      mbar_init(bar(st.item_empty[x]), 8 + 2);  // softmax warps and both issuers
      mbar_init(bar(st.drain[x]), 1);
    }
    mbar_init(bar(st.never), 1);
    st.abort_flag = 0;
    if (kSelfTest) st.t_start = global_timer_ns();
    fence_barrier_init();
  }
  if (warp == kTcSWarp) {
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
    uint32_t k_issued = 0, v_issued = 0, q_issued = 0;  // copies issued so far, per ring
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
      q_issued = i + 1;
      bool ok = true;
      constexpr int kPagesPerBlock = kTcKeys / kPage;  // 8: four blocks per 32-page chunk
      // K of block b, then V of block b - 1 (same pool rows, kept from the
      // previous iteration); V of the last block after the loop
      int y_prev[kPagesPerBlock];
      auto load_block = [&](bool is_k, uint32_t it, const int (&y)[kPagesPerBlock]) -> bool {
        const int nst = is_k ? kTcKStages : kTcVStages;
        const int s = it % nst;
        uint64_t* full = is_k ? st.k_full : st.v_full;
        uint64_t* empty = is_k ? st.k_empty : st.v_empty;
        if (it >= (uint32_t)nst &&
            !__all_sync(0xffffffffu, wait_bar(bar(empty[s]), ((it / nst) - 1) & 1, abort_flag)))
          return false;
        if (lane == 0) {
          const uint32_t dst = (is_k ? sK : sV) + s * kTcKvBytes;
          mbar_arrive_expect_tx(bar(full[s]), kTcKvBytes);
#pragma unroll
          for (int j = 0; j < kPagesPerBlock; ++j)
            tma_load_2d(dst + j * kTileBytes, is_k ? &kmap : &vmap, 0, y[j], bar(full[s]), pol);
        }
        (is_k ? k_issued : v_issued) = it + 1;
        return true;
      };
      for (int b = 0; b < nb; ++b, ++kv_it) {
        if (kSelfTest && p.selftest_stall == 1 && i == 0 && b == 1) {
          if (lane == 0) selftest_stall(bar(st.never), &st.abort_flag);
          __syncwarp();
          ok = false;
          break;
        }
        if (b > 0 && (b * kPagesPerBlock) % 32 == 0) {
          pid_cur = pid_next;
          pid_next = load_chunk(b * kPagesPerBlock / 32 + 1);
        }
        const int lane0 = (b * kPagesPerBlock) % 32;
        int y[kPagesPerBlock];
#pragma unroll
        for (int j = 0; j < kPagesPerBlock; ++j) {
          const int pid = __shfl_sync(0xffffffffu, pid_cur, lane0 + j);
          y[j] = pid < 0 ? p.oob_row : (pid * Hkv + kvh) * kPage;
        }
        if (!load_block(true, kv_it, y) || (b > 0 && !load_block(false, kv_it - 1, y_prev))) {
          ok = false;
          break;
        }
#pragma unroll
        for (int j = 0; j < kPagesPerBlock; ++j) y_prev[j] = y[j];
      }
      if (ok && nb > 0 && !load_block(false, kv_it - 1, y_prev)) ok = false;
      if (!ok) break;
    }
    // After an abort, copies may still be in flight into the rings: wait
    // (bounded) for the last ones issued to each ring before the CTA ends.
    // Each such copy is the latest of its stage, so its full barrier's phase
    // parity identifies it. A finished kernel has none in flight.
    if (*abort_flag && lane == 0) {
      for (uint32_t it = k_issued > (uint32_t)kTcKStages ? k_issued - kTcKStages : 0; it < k_issued; ++it)
        mbar_wait(bar(st.k_full[it % kTcKStages]), (it / kTcKStages) & 1);
      for (uint32_t it = v_issued > (uint32_t)kTcVStages ? v_issued - kTcVStages : 0; it < v_issued; ++it)
        mbar_wait(bar(st.v_full[it % kTcVStages]), (it / kTcVStages) & 1);
      if (q_issued > 0) mbar_wait(bar(st.q_full), (q_issued - 1) & 1);
    }
  } else if (warp == kTcSWarp || warp == kTcPvWarp) {
    // ---------------------------------------------------------- MMA issuers
    // One issuing warp per tile (warp 9: tile A, warp 10: tile B), each in
    // its tile's own order S(b), PV(b - 1), so that neither tile's MMAs wait
    // behind the other tile's softmax. The whole warp runs the loop in step
    // and one elected lane issues each MMA: operands computed by a lone lane
    // of a diverged warp leave the uniform datapath, which costs each MMA
    // about 50 cycles of issue (a 128 x 64 x 16 MMA computes in 32; the PV
    // issue of a block went 717 -> 474 cycles). Their MMAs touch disjoint TMEM and are
    // ordered only through the mbarriers; a K or V stage and the query tiles
    // are released by two commits, one per tile. The loops are lean:
    // descriptors are computed once and stepped by constants (the
    // start-address field counts 16-byte units and cannot overflow: shared
    // memory ends below 256 KiB).
    {
      constexpr uint32_t idS = idesc_bf16(kTcRows, kTcKeys, false, false);
      constexpr uint32_t idO = idesc_bf16(kTcRows, kHeadDim, false, true);
      constexpr uint64_t kStageStep = kTcKvBytes / 16, kVStep = 16 * kRowBytes / 16;
      const uint64_t kdesc0 = smem_desc_sw128(sK, 16, 1024);
      const uint64_t vdesc0 = smem_desc_sw128(sV, 1024, 1024);
      // issuer x drives tile x: S_x(b) as soon as K(b) and its S buffer are
      // free, then O_x += P_x(b - 1) V(b - 1) once that P is ready; the two
      // tiles never wait on each other's softmax
      const int x = warp == kTcSWarp ? 0 : 1;
      const uint32_t scol = tmem + col_s(x), pcol = tmem + col_p(x), ocol = tmem + col_o(x);
      const uint64_t qd = smem_desc_sw128(sQ + x * kTcTileQBytes, 16, 1024);
      uint32_t blk = 0;
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
        for (int b = 0; b <= nb && ok; ++b) {
          if (kSelfTest && p.selftest_stall == 2 && x == 0 && i == 0 && b == 1) {
            selftest_stall(bar(st.never), &st.abort_flag);
            ok = false;
            break;
          }
          if (b < nb) {  // S_x(b)
            const uint32_t bk = blk + b;
            const int s = bk % kTcKStages;
            // S buffer x was last loaded by the softmax of block bk - 1
            if (!wait_bar(bar(st.k_full[s]), (bk / kTcKStages) & 1, abort_flag) ||
                (bk >= 1 && !wait_bar(bar(st.s_free[x]), (bk - 1) & 1, abort_flag))) {
              ok = false;
              break;
            }
            tc_fence_after();
            const uint64_t kd = kdesc0 + s * kStageStep;
            tc_mma_ss_e(scol, qd, kd, idS, 0u);
#pragma unroll
            for (int kk = 1; kk < kHeadDim / 16; ++kk)
              tc_mma_ss_e(scol, qd + (uint64_t)(kk * 2), kd + (uint64_t)(kk * 2), idS, 1u);
            tc_commit_e(bar(st.s_full[x]));
            tc_commit_e(bar(st.k_empty[s]));              // released when both tiles have read it
            if (b == nb - 1) tc_commit_e(bar(st.q_empty));  // likewise
          }
          if (b >= 1) {  // O_x += P_x(b - 1) V(b - 1)
            const uint32_t bv = blk + b - 1;
            const int sv = bv % kTcVStages;
            if (!wait_bar(bar(st.v_full[sv]), (bv / kTcVStages) & 1, abort_flag) ||
                !wait_bar(bar(st.p_full[x]), bv & 1, abort_flag) ||
                (b == 1 && i >= 1 && !wait_bar(bar(st.o_free[x]), (i - 1) & 1, abort_flag))) {
              ok = false;
              break;
            }
            tc_fence_after();
            const uint64_t vd = vdesc0 + sv * kStageStep;
            tc_mma_ts_e(ocol, pcol, vd, idO, b > 1 ? 1u : 0u);
#pragma unroll
            for (int kk = 1; kk < kTcKeys / 16; ++kk) tc_mma_ts_e(ocol, pcol + kk * 8, vd + kk * kVStep, idO, 1u);
            tc_commit_e(bar(st.o_ready[x]));
            tc_commit_e(bar(st.v_empty[sv]));  // released when both tiles have read it
          }
        }
        if (!ok) break;
        blk += nb;
        if (lane == 0) mbar_arrive(bar(st.item_empty[slot]));
      }
      // wait for this thread's MMAs still in flight (only after an abort can
      // any be), so that TMEM is not freed under them
      tc_commit_e(bar(st.drain[x]));
      mbar_wait(bar(st.drain[x]), 0);
    }
  } else {
    // ------------------------------------------------------------- softmax
    const int x = warp >> 2;                      // tile A (0) or B (1)
    const int row = threadIdx.x & (kTcRows - 1);  // TMEM lane
    const int wq = warp & 3;
    const uint32_t lane_off = (uint32_t)(wq * 32) << 16;
    const uint32_t cS = tmem + lane_off + col_s(x), cP = tmem + lane_off + col_p(x), cO = tmem + lane_off + col_o(x);
    const int tile_tok = kTcRows / g;
    uint32_t blk = 0;
    bool ok = true;
    for (int i = 0; ok; ++i) {
      const int slot = i & 1;
      ok = __all_sync(0xffffffffu, wait_bar_poll(bar(st.item_full[slot]), (i >> 1) & 1, abort_flag));
      if (!ok) break;
      const int idx = st.item_idx[slot];
      const AppendItem a = st.items[slot];
      if (idx >= n_items) break;
      const int kvh = idx % Hkv;
      const int tok = x * tile_tok + row / g, head = row % g;
      const bool valid = tok < a.n_tok;
      const int last_tok = max(a.n_tok - 1, 0);
      const int pos = a.pos_begin + min(tok, last_tok);
      const int lo = p.window > 0 ? pos - p.window + 1 : 0;
      const int kb0 = (a.key_begin / kPage) * kPage;
      const int nb = (a.key_end - kb0 + kTcKeys - 1) / kTcKeys;
      // warp-uniform position range of this warp's rows, for mask skipping
      const int wp_min = a.pos_begin + min(x * tile_tok + (wq * 32) / g, last_tok);
      const int wp_max = a.pos_begin + min(x * tile_tok + (wq * 32 + 31) / g, last_tok);
      float m_ref = -INFINITY, l = 0.f;
      for (int b = 0; b < nb; ++b, ++blk) {
        if (kSelfTest && p.selftest_stall == 0 && x == 0 && i == 0 && b == 1) {
          if (lane == 0) selftest_stall(bar(st.never), &st.abort_flag);
          __syncwarp();
          ok = false;
          break;
        }
        ok = __all_sync(0xffffffffu, wait_bar_poll(bar(st.s_full[x]), blk & 1, abort_flag));
        if (!ok) break;
        tc_fence_after();
        const int kb = kb0 + b * kTcKeys;
        uint32_t sv[2][32], pk[32];
        // ---- chunk 0: keys kb .. kb + 63
        tmem_ld32(cS, sv[0]);
        tmem_ld32(cS + 32, sv[1]);
        tmem_ld_wait();
        if ((kb + 63 > wp_min) || (p.window > 0 && kb < wp_max - p.window + 1)) mask_chunk(sv, kb, pos, lo);
        float alpha = 1.f;
        float l0 = chunk_probs(sv, p.scale_log2, m_ref, alpha, pk);
        // the single P buffer was last read by PV_X(blk - 1)
        if (blk >= 1) {
          ok = __all_sync(0xffffffffu, wait_bar_poll(bar(st.o_ready[x]), (blk - 1) & 1, abort_flag));
          if (!ok) break;
          tc_fence_after();
        }
        tmem_st32(cP, pk);
        // ---- chunk 1: keys kb + 64 .. kb + 127; then S_X is free
        tmem_ld32(cS + 64, sv[0]);
        tmem_ld32(cS + 96, sv[1]);
        tmem_ld_wait();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(bar(st.s_free[x]));
        if ((kb + 127 > wp_min) || (p.window > 0 && kb + 64 < wp_max - p.window + 1)) mask_chunk(sv, kb + 64, pos, lo);
        float a1 = 1.f;
        const float l1 = chunk_probs(sv, p.scale_log2, m_ref, a1, pk);
        if (__any_sync(0xffffffffu, a1 != 1.f)) {
          // rare: the reference rose inside the block; rescale chunk 0's P too
          tmem_st_wait();
          uint32_t pv[32];
          tmem_ld32(cP, pv);
          tmem_ld_wait();
#pragma unroll
          for (int e = 0; e < 32; ++e) {
            const float2 f = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&pv[e]));
            pv[e] = pack_bf16x2(f.x * a1, f.y * a1);
          }
          tmem_st32(cP, pv);
          l0 *= a1;
          alpha *= a1;
        }
        tmem_st32(cP + 32, pk);
        l = l * alpha + (l0 + l1);
        // V rows of slots no query of the item sees (before key_begin on the
        // partial first page of a window, from key_end on the partial last
        // page) were perhaps never written and may hold NaN, which a zero
        // weight does not cancel (0 x NaN = NaN). Once the block's V stage
        // has landed they are zeroed in shared memory (at most 15 rows each;
        // whole pages past the row's end arrive as zeros already), then
        // handed to the async proxy before this tile's PV may read them. Both
        // tiles' warps write the same zeros, each before its own p_full.
        {
          const bool lo_edge = b == 0 && kb0 < a.key_begin;
          const bool hi_edge = b == nb - 1 && (a.key_end & (kPage - 1)) != 0;
          if (lo_edge || hi_edge) {
            const uint32_t sv_i = blk % kTcVStages;
            ok = __all_sync(0xffffffffu, wait_bar_poll(bar(st.v_full[sv_i]), (blk / kTcVStages) & 1, abort_flag));
            if (!ok) break;
            const uint32_t vst = sV + sv_i * kTcKvBytes;
            const int zr = row >> 3, zc = row & 7;  // key row (0..15) and 16-byte chunk of this thread
            if (lo_edge && zr < a.key_begin - kb0) st_shared_zero16(vst + zr * kRowBytes + zc * 16);
            if (hi_edge) {
              const int r0 = a.key_end - kb;  // first row past the row's end, inside this block
              if (zr < kPage - (r0 & (kPage - 1))) st_shared_zero16(vst + (r0 + zr) * kRowBytes + zc * 16);
            }
            fence_proxy_async();
          }
        }
        // O_X may only be rescaled once PV_X(blk - 1) has completed (waited above)
        if (b > 0 && __any_sync(0xffffffffu, alpha != 1.f)) {
          uint32_t ov[32];
#pragma unroll
          for (int h = 0; h < 2; ++h) {
            tmem_ld32(cO + 32 * h, ov);
            tmem_ld_wait();
#pragma unroll
            for (int e = 0; e < 32; ++e) ov[e] = __float_as_uint(__uint_as_float(ov[e]) * alpha);
            tmem_st32(cO + 32 * h, ov);
          }
        }
        tmem_st_wait();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(bar(st.p_full[x]));
      }
      if (!ok) break;
      // epilogue: the last PV_X of the item
      if (nb > 0) {
        ok = __all_sync(0xffffffffu, wait_bar_poll(bar(st.o_ready[x]), (blk - 1) & 1, abort_flag));
        if (!ok) break;
      }
      tc_fence_after();
      uint32_t ov[2][32];
      tmem_ld32(cO, ov[0]);
      tmem_ld32(cO + 32, ov[1]);
      tmem_ld_wait();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) {
        mbar_arrive(bar(st.o_free[x]));
        mbar_arrive(bar(st.item_empty[slot]));
      }
      if constexpr (kOutHost) {
        // O / l as bf16, this thread's row in 32 words (dims 2j, 2j + 1),
        // written as four 32-byte pieces (whole sectors) when out is 32-byte
        // aligned, else eight 16-byte ones
        float inv = l > 0.f ? 1.f / l : 0.f;
        float lse2 = l > 0.f ? m_ref + __log2f(l) : -INFINITY;
        if (p.sinks != nullptr) inv = finish_with_sink(m_ref, l, sink_log2(p, kvh * g + head), &lse2);
        if (valid) {
          uint32_t w[32];
#pragma unroll
          for (int j = 0; j < 32; ++j)
            w[j] = pack_bf16x2(__uint_as_float(ov[j >> 4][2 * (j & 15)]) * inv,
                               __uint_as_float(ov[j >> 4][2 * (j & 15) + 1]) * inv);
          const size_t orow = (size_t)(a.token_begin + tok) * Hq + kvh * g + head;
          uint8_t* dst = reinterpret_cast<uint8_t*>(p.out + orow * kHeadDim);
          if ((reinterpret_cast<uintptr_t>(p.out) & 31) == 0) {
#pragma unroll
            for (int q = 0; q < 4; ++q) st_global_v8(dst + 32 * q, w + 8 * q);
          } else {
#pragma unroll
            for (int q = 0; q < 8; ++q)
              reinterpret_cast<uint4*>(dst)[q] = make_uint4(w[4 * q], w[4 * q + 1], w[4 * q + 2], w[4 * q + 3]);
          }
          p.lse[orow] = lse2 * 0.69314718055994531f;
        }
      } else if (valid) {
        float inv = l > 0.f ? 1.f / l : 0.f;
        float lse2 = l > 0.f ? m_ref + __log2f(l) : -INFINITY;
        if (p.sinks != nullptr) inv = finish_with_sink(m_ref, l, sink_log2(p, kvh * g + head), &lse2);
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
        p.lse[orow] = lse2 * 0.69314718055994531f;
      }
    }
  }

  // every role ends here; a timed-out role has set the abort flag
  __syncwarp();
  if (kSelfTest && lane == 0 && blockIdx.x == 0) p.selftest_report[1 + warp] = (int64_t)(global_timer_ns() - st.t_start);
  if (threadIdx.x == 0 && *abort_flag) raise_status(p, kStatusTimeout);
  tc_fence_before();
  __syncthreads();
  if (warp == kTcSWarp) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
    if (kSelfTest && lane == 0 && blockIdx.x == 0) {
      p.selftest_report[0] = *abort_flag;
      p.selftest_report[12] = (int64_t)kSelftestStallNs;
      p.selftest_report[13] = (int64_t)kWaitTimeoutNs;
      p.selftest_report[14] = 1;  // TMEM freed
    }
  }
}

// out_host: p.out is page-locked host memory (the form that writes whole sectors).
cudaError_t launch_append_tc(const CUtensorMap& kmap, const CUtensorMap& vmap, const CUtensorMap& qmap,
                             const AttnParams& p, int grid, bool out_host, cudaStream_t stream) {
  if (out_host)
    append_tc_kernel<false, true><<<grid, kTcThreads, append_tc_smem_bytes(), stream>>>(kmap, vmap, qmap, p);
  else
    append_tc_kernel<false, false><<<grid, kTcThreads, append_tc_smem_bytes(), stream>>>(kmap, vmap, qmap, p);
  return cudaGetLastError();
}

// The self-test form: one CTA, p.selftest_stall names the stalled role and
// p.selftest_report receives the abort flag and each warp's exit time.
cudaError_t launch_append_tc_selftest(const CUtensorMap& kmap, const CUtensorMap& vmap, const CUtensorMap& qmap,
                                      const AttnParams& p, cudaStream_t stream) {
  append_tc_kernel<true, false><<<1, kTcThreads, append_tc_smem_bytes(), stream>>>(kmap, vmap, qmap, p);
  return cudaGetLastError();
}

cudaError_t prepare_append_tc_kernel(int* blocks_per_sm) {
  for (auto fn : {append_tc_kernel<false, false>, append_tc_kernel<true, false>, append_tc_kernel<false, true>}) {
    cudaError_t e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)append_tc_smem_bytes());
    if (e != cudaSuccess) return e;
    e = cudaFuncSetAttribute(fn, cudaFuncAttributePreferredSharedMemoryCarveout, cudaSharedmemCarveoutMaxShared);
    if (e != cudaSuccess) return e;
  }
  return cudaOccupancyMaxActiveBlocksPerMultiprocessor(blocks_per_sm, append_tc_kernel<false, false>, kTcThreads,
                                                       append_tc_smem_bytes());
}

}  // namespace mcpu
