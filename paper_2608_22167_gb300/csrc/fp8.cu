// fp8 (e4m3) KV pages: the quantizing KV append and the split-KV decode /
// cascade kernel that reads them (a storage variant; the paper keeps bf16).
//
// Storage, per (page, kv head) block:
//   k8  [16 keys][64 dims]  e4m3 codes, row-major (1 KiB)
//   v8  [64 dims][16 keys]  e4m3 codes, TRANSPOSED (1 KiB)
//   k_scale, v_scale [16]   float, one scale per (token, kv head) row
// Each new row x (64 bf16) is stored as a = max|x_i|, scale = a / 448 and
// code_i = e4m3(x_i * (448 / a)) (round to nearest even, saturating), in
// float arithmetic; an all-zero row stores zeros. A key is code * scale.
//
// Decode over fp8 pages follows the bf16 kernel (one warp per work item,
// a per-warp ring of pages, m16n8k16 tensor-core tiles, online softmax,
// partials merged by log-sum-exp) with these differences:
//   - a page's 2 KiB of codes and 128 B of scales arrive by four untiled
//     bulk copies (no tensor map), 2176 bytes per (page, kv head);
//   - codes become fp16 operands by integer ops: an e4m3 code c placed in
//     the high byte of a 16-bit lane gives ((c & 0x7f) << 7) | sign, the
//     fp16 whose value is exactly value(c) * 2^-8 (subnormals included), so
//     both products run as f16 x f16 -> f32;
//   - q enters as fp16 times a power of two per query vector (its largest
//     entry lands in [2^14, 2^15)); the key scale, that power of two and
//     the softmax scale multiply each score in fp32;
//   - P . V takes P' = p * v_scale * 2^8 * 2^F in fp16, F a per-item power
//     of two that only decreases (the page's largest v_scale sets it, so P'
//     stays below 2^15); the accumulator is rescaled when F drops and
//     divided by 2^F at the end.
// Which dims/keys meet in one MMA k-slot is a permutation chosen so that
// every operand comes from a 32- or 128-bit shared-memory load: row 2r and
// 2r + 1 of the K block and word c (keys 4c..4c+3) of the transposed V rows.
#include <cuda_fp16.h>

#include "common.cuh"

namespace mcpu {

constexpr int kF8Warps = 4;
constexpr int kF8Stages = 8;
constexpr int kF8Block = kPage * kHeadDim;                      // codes of one block: 1 KiB
constexpr int kF8ScaleBytes = kPage * 4;                        // 64
constexpr int kF8StageBytes = 2 * kF8Block + 2 * kF8ScaleBytes;  // 2176
constexpr int kF8RingBytes = kF8Stages * kF8StageBytes;

struct F8Pools {
  const uint8_t* k8;
  const uint8_t* v8;
  const float* k_scale;
  const float* v_scale;
};

size_t decode_fp8_smem_bytes() {
  return 128 /* alignment slack */ + (size_t)kF8Warps * kF8RingBytes + (size_t)kF8Warps * kF8Stages * 8;
}

// Two e4m3 codes in bits 8..15 and 24..31 of y -> f16x2 of value(code) * 2^-8.
__device__ __forceinline__ uint32_t e4m3_pair_to_f16x2(uint32_t y) {
  return ((y >> 1) & 0x3F803F80u) | (y & 0x80008000u);
}

__device__ __forceinline__ uint32_t pack_f16x2(float lo, float hi) {
  __half2 v = __floats2half2_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}

// 2^e as a float for -126 <= e <= 127
__device__ __forceinline__ float exp2i(int e) { return __uint_as_float((uint32_t)(e + 127) << 23); }

// floor(log2(x)) of a positive finite float (subnormals give -127)
__device__ __forceinline__ int ilog2f(float x) { return (int)((__float_as_uint(x) >> 23) & 0xFF) - 127; }

template <int NT>
__global__ void __launch_bounds__(kF8Warps * 32) decode_fp8_kernel(const F8Pools pools, const AttnParams p) {
  extern __shared__ uint8_t smem_raw[];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int r = lane >> 2, c = lane & 3;
  const uint32_t raw = smem_addr(smem_raw);
  const uint32_t base = (raw + 127u) & ~127u;
  const uint32_t ring = base + warp * kF8RingBytes;
  const uint32_t bars = base + kF8Warps * kF8RingBytes + warp * kF8Stages * 8;
  uint8_t* ring_ptr = smem_raw + (ring - raw);
  float* scratch = reinterpret_cast<float*>(ring_ptr);

  if (lane == 0) {
    for (int s = 0; s < kF8Stages; ++s) mbar_init(bars + 8 * s, 1);
    fence_barrier_init();
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
      const CascadeItem ci = citems[rec];
      row = ci.first_row;
      pb = ci.page_begin;
      pe = ci.page_end;
      member_off = ci.member_off;
      n_members = ci.n_members;
      split = ci.split;
    }
    const int* bt_row = p.block_table + (size_t)row * p.max_pages;

    // Query vector r (+ 8 nt) as the B operand: this lane holds its dims
    // 16c .. 16c + 15 times 2^eq; k-slot 2c + e of step kk is dim
    // 16c + 4kk + 2e, k-slot 2c + 8 + e is dim 16c + 4kk + 1 + 2e.
    uint32_t qb[NT][4][2];
    float qm[NT][2];  // score factor of query vectors 2c and 2c + 1
#pragma unroll
    for (int nt = 0; nt < NT; ++nt) {
      const int qv = nt * 8 + r;
      int tok = -1, head = 0;
      if (NT == 1) {
        if (qv < g) tok = token, head = kvh * g + qv;
      } else {
        const int m = qv / g;
        if (m < n_members) tok = members[member_off + m].token, head = kvh * g + qv % g;
      }
      float x[16];
      if (tok >= 0) {
        const uint4* qp = reinterpret_cast<const uint4*>(p.q + ((size_t)tok * Hq + head) * kHeadDim) + 2 * c;
        const uint4 u0 = __ldg(qp), u1 = __ldg(qp + 1);
        const uint32_t w[8] = {u0.x, u0.y, u0.z, u0.w, u1.x, u1.y, u1.z, u1.w};
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          x[2 * i] = __uint_as_float(w[i] << 16);
          x[2 * i + 1] = __uint_as_float(w[i] & 0xFFFF0000u);
        }
      } else {
#pragma unroll
        for (int i = 0; i < 16; ++i) x[i] = 0.f;
      }
      float mx = 0.f;
#pragma unroll
      for (int i = 0; i < 16; ++i) mx = fmaxf(mx, fabsf(x[i]));
      mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 1));
      mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 2));
      int eq = mx > 0.f ? 14 - ilog2f(mx) : 0;
      eq = min(max(eq, -126), 126);
      const float up = exp2i(eq);
      const float my_qm = exp2i(-eq) * 256.f * p.scale_log2;
#pragma unroll
      for (int kk = 0; kk < 4; ++kk) {
        qb[nt][kk][0] = pack_f16x2(x[4 * kk] * up, x[4 * kk + 2] * up);
        qb[nt][kk][1] = pack_f16x2(x[4 * kk + 1] * up, x[4 * kk + 3] * up);
      }
      qm[nt][0] = __shfl_sync(0xffffffffu, my_qm, (2 * c) * 4);
      qm[nt][1] = __shfl_sync(0xffffffffu, my_qm, (2 * c + 1) * 4);
    }

    // Page ids: lane i caches the id of page (chunk + i); lane 0 issues.
    const int n = pe - pb;
    int chunk_base = -32, pid_reg = 0;
    uint32_t bad_stages = 0;  // stages holding an invalid page (warp-uniform)
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
      const uint32_t s = (seq + k) % kF8Stages;
      bad_stages = pid < 0 ? (bad_stages | (1u << s)) : (bad_stages & ~(1u << s));
      if (lane == 0) {
        const uint32_t bar = bars + 8 * s;
        if (pid < 0) {
          mbar_arrive(bar);  // nothing to copy: the page's keys are masked
        } else {
          const size_t blk = (size_t)pid * Hkv + kvh;
          const uint32_t dst = ring + s * kF8StageBytes;
          mbar_arrive_expect_tx(bar, kF8StageBytes);
          bulk_load(dst, pools.k8 + blk * kF8Block, kF8Block, bar, pol);
          bulk_load(dst + kF8Block, pools.v8 + blk * kF8Block, kF8Block, bar, pol);
          bulk_load(dst + 2 * kF8Block, pools.k_scale + blk * kPage, kF8ScaleBytes, bar, pol);
          bulk_load(dst + 2 * kF8Block + kF8ScaleBytes, pools.v_scale + blk * kPage, kF8ScaleBytes, bar, pol);
        }
      }
    };
    const int pre = n < kF8Stages ? n : kF8Stages;
    for (int k = 0; k < pre; ++k) issue(k);

    float m_run[NT][2], l_run[NT][2], acc[4][NT][4];
#pragma unroll
    for (int nt = 0; nt < NT; ++nt) {
      m_run[nt][0] = m_run[nt][1] = -INFINITY;
      l_run[nt][0] = l_run[nt][1] = 0.f;
#pragma unroll
      for (int mt = 0; mt < 4; ++mt)
#pragma unroll
        for (int e = 0; e < 4; ++e) acc[mt][nt][e] = 0.f;
    }
    int F = 120;  // P' = p * v_scale * 2^8 * 2^F; acc is held in units of 2^F

    bool timed_out = false;
    for (int k = 0; k < n; ++k) {
      const uint32_t s = (seq + k) % kF8Stages;
      const uint32_t phase = ((seq + k) / kF8Stages) & 1u;
      const bool ok = __any_sync(0xffffffffu, mbar_wait(bars + 8 * s, phase));
      if (!ok) {
        timed_out = true;
        break;
      }
      const uint8_t* st = ring_ptr + s * kF8StageBytes;
      const uint4 KA = *reinterpret_cast<const uint4*>(st + (2 * r) * kHeadDim + 16 * c);
      const uint4 KB = *reinterpret_cast<const uint4*>(st + (2 * r + 1) * kHeadDim + 16 * c);
      const float2 ks = *reinterpret_cast<const float2*>(st + 2 * kF8Block + 8 * r);
      const float2 vs = *reinterpret_cast<const float2*>(st + 2 * kF8Block + kF8ScaleBytes + 8 * r);

      // S^T[16 keys x 8*NT query vectors]: M row r is key 2r, row r + 8 key 2r + 1
      float cc[NT][4];
#pragma unroll
      for (int nt = 0; nt < NT; ++nt) cc[nt][0] = cc[nt][1] = cc[nt][2] = cc[nt][3] = 0.f;
      {
        const uint32_t wa[4] = {KA.x, KA.y, KA.z, KA.w}, wb[4] = {KB.x, KB.y, KB.z, KB.w};
#pragma unroll
        for (int kk = 0; kk < 4; ++kk) {
          const uint32_t a0 = e4m3_pair_to_f16x2(wa[kk] << 8), a1 = e4m3_pair_to_f16x2(wb[kk] << 8);
          const uint32_t a2 = e4m3_pair_to_f16x2(wa[kk]), a3 = e4m3_pair_to_f16x2(wb[kk]);
#pragma unroll
          for (int nt = 0; nt < NT; ++nt) mma_f16_16816(cc[nt], a0, a1, a2, a3, qb[nt][kk][0], qb[nt][kk][1]);
        }
      }

      // keys outside [first_key, seq_len) or on an invalid page are masked
      const int j0 = (pb + k) * kPage + 2 * r;
      const bool page_ok = ((bad_stages >> s) & 1u) == 0;
      bool v0 = page_ok, v1 = page_ok;
      if (NT == 1) {
        v0 = v0 && j0 >= first_key && j0 < seq_len;
        v1 = v1 && (j0 + 1) >= first_key && (j0 + 1) < seq_len;
      }
      // the page's power of two for P' (F only decreases)
      const float u0 = v0 ? vs.x * 256.f : 0.f, u1 = v1 ? vs.y * 256.f : 0.f;
      float umax = fmaxf(u0, u1);
      umax = fmaxf(umax, __shfl_xor_sync(0xffffffffu, umax, 4));
      umax = fmaxf(umax, __shfl_xor_sync(0xffffffffu, umax, 8));
      umax = fmaxf(umax, __shfl_xor_sync(0xffffffffu, umax, 16));
      int F_new = F;
      if (umax > 0.f) F_new = min(F, max(14 - ilog2f(umax), -120));
      const float dF = F_new < F ? (F_new - F >= -126 ? exp2i(F_new - F) : 0.f) : 1.f;
      F = F_new;
      const float pf = exp2i(F);
      const float w0 = u0 * pf, w1 = u1 * pf;

      uint32_t pb0[NT], pb1[NT];
#pragma unroll
      for (int nt = 0; nt < NT; ++nt) {
        const float s00 = v0 ? cc[nt][0] * ks.x * qm[nt][0] : -INFINITY;
        const float s01 = v0 ? cc[nt][1] * ks.x * qm[nt][1] : -INFINITY;
        const float s10 = v1 ? cc[nt][2] * ks.y * qm[nt][0] : -INFINITY;
        const float s11 = v1 ? cc[nt][3] * ks.y * qm[nt][1] : -INFINITY;
        float mx0 = fmaxf(s00, s10), mx1 = fmaxf(s01, s11);
#pragma unroll
        for (int o = 4; o < 32; o <<= 1) {
          mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, o));
          mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, o));
        }
        const float mn0 = fmaxf(m_run[nt][0], mx0), mn1 = fmaxf(m_run[nt][1], mx1);
        const float mu0 = mn0 == -INFINITY ? 0.f : mn0;
        const float mu1 = mn1 == -INFINITY ? 0.f : mn1;
        const float al0 = fast_exp2(m_run[nt][0] - mu0), al1 = fast_exp2(m_run[nt][1] - mu1);
        const float p00 = fast_exp2(s00 - mu0), p10 = fast_exp2(s10 - mu0);
        const float p01 = fast_exp2(s01 - mu1), p11 = fast_exp2(s11 - mu1);
        l_run[nt][0] = l_run[nt][0] * al0 + p00 + p10;
        l_run[nt][1] = l_run[nt][1] * al1 + p01 + p11;
        m_run[nt][0] = mn0;
        m_run[nt][1] = mn1;
        const float ac0 = al0 * dF, ac1 = al1 * dF;
#pragma unroll
        for (int mt = 0; mt < 4; ++mt) {
          acc[mt][nt][0] *= ac0;
          acc[mt][nt][1] *= ac1;
          acc[mt][nt][2] *= ac0;
          acc[mt][nt][3] *= ac1;
        }
        pb0[nt] = movmatrix_trans(pack_f16x2(p00 * w0, p01 * w0));
        pb1[nt] = movmatrix_trans(pack_f16x2(p10 * w1, p11 * w1));
      }

      // O^T[64 dims x 8*NT] += V^T P'^T: k-slot 2c + e is key 4c + 2e,
      // k-slot 2c + 8 + e is key 4c + 1 + 2e (word c of a transposed V row)
#pragma unroll
      for (int mt = 0; mt < 4; ++mt) {
        const uint32_t x0 = *reinterpret_cast<const uint32_t*>(st + kF8Block + (16 * mt + r) * kPage + 4 * c);
        const uint32_t x1 = *reinterpret_cast<const uint32_t*>(st + kF8Block + (16 * mt + r + 8) * kPage + 4 * c);
        const uint32_t a0 = e4m3_pair_to_f16x2(x0 << 8), a1 = e4m3_pair_to_f16x2(x1 << 8);
        const uint32_t a2 = e4m3_pair_to_f16x2(x0), a3 = e4m3_pair_to_f16x2(x1);
#pragma unroll
        for (int nt = 0; nt < NT; ++nt) mma_f16_16816(acc[mt][nt], a0, a1, a2, a3, pb0[nt], pb1[nt]);
      }

      // release the stage to the async proxy, then refill it
      fence_proxy_async();
      __syncwarp();
      if (k + kF8Stages < n) issue(k + kF8Stages);
    }

    if (timed_out) {
      raise_status(p, kStatusTimeout);
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
    const float unit = F >= -126 ? exp2i(-F) : 0.f;  // acc -> output units (F <= 120)
    constexpr int kLd = kHeadDim + 1;
    float* so = scratch;                 // [8*NT][kLd]
    float* sl = scratch + 8 * NT * kLd;  // [8*NT] base-2 lse
#pragma unroll
    for (int nt = 0; nt < NT; ++nt) {
#pragma unroll
      for (int e = 0; e < 2; ++e) {
        const int qv = nt * 8 + 2 * c + e;
        const float l = l_run[nt][e];
        float inv = l > 0.f ? 1.f / l : 0.f;
        float lse2 = l > 0.f ? m_run[nt][e] + __log2f(l) : -INFINITY;
        if (NT == 1 && p.sinks != nullptr && slot < 0 && qv < g)
          inv = finish_with_sink(m_run[nt][e], l, sink_log2(p, kvh * g + qv), &lse2);
        inv *= unit;
#pragma unroll
        for (int mt = 0; mt < 4; ++mt) {
          so[qv * kLd + mt * 16 + r] = acc[mt][nt][e] * inv;
          so[qv * kLd + mt * 16 + r + 8] = acc[mt][nt][e + 2] * inv;
        }
        if (r == 0) sl[qv] = lse2;
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
    // the staging area is the copy ring: order these generic accesses
    // before the next item's async-proxy writes
    fence_proxy_async();
    __syncwarp();
  }
}

// ------------------------------------------------------------ fp8 KV append

constexpr int kF8AppendWarps = 8;

struct F8AppendParams {
  const __nv_bfloat16* k_new;  // [T, Hkv, D]
  const __nv_bfloat16* v_new;
  uint8_t* k8;                 // [P, Hkv, 16, D]
  uint8_t* v8;                 // [P, Hkv, D, 16]
  float* k_scale;              // [P, Hkv, 16]
  float* v_scale;
  const int32_t* block_table;
  const int32_t* seq_lens;
  const int32_t* qsl;
  int32_t* status;
  int32_t num_seqs, total_q, max_pages, num_pages, num_kv_heads;
};

// The e4m3 codes of x0 (low byte) and x1 (high byte): nearest, ties to
// even, saturating at +-448.
__device__ __forceinline__ uint32_t e4m3x2(float x0, float x1) {
  uint16_t d;
  asm("cvt.rn.satfinite.e4m3x2.f32 %0, %1, %2;" : "=h"(d) : "f"(x1), "f"(x0));
  return d;
}

// one warp per (token, kv head): lane l quantizes dims 2l and 2l + 1 of K and V
__global__ void __launch_bounds__(kF8AppendWarps * 32) kv_append_fp8_kernel(const F8AppendParams p) {
  const int lane = threadIdx.x & 31;
  const int w = blockIdx.x * kF8AppendWarps + (threadIdx.x >> 5);
  if (w >= p.total_q * p.num_kv_heads) return;
  const int t = w / p.num_kv_heads, h = w % p.num_kv_heads;
  int dst = -1;
  if (lane == 0) {
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
        const int pos = S - L + (t - q0);
        const int page = __ldg(p.block_table + (size_t)lo * p.max_pages + pos / kPage);
        if (page < 0 || page >= p.num_pages)
          atomicOr(p.status, kStatusBadPage);
        else
          dst = page * kPage + pos % kPage;
      }
    }
  }
  dst = __shfl_sync(0xffffffffu, dst, 0);
  if (dst < 0) return;
  const int page = dst / kPage, slot = dst % kPage;
  const size_t blk = (size_t)page * p.num_kv_heads + h;
#pragma unroll
  for (int which = 0; which < 2; ++which) {
    const __nv_bfloat16* src = (which ? p.v_new : p.k_new) + ((size_t)t * p.num_kv_heads + h) * kHeadDim;
    const uint32_t bits = __ldg(reinterpret_cast<const uint32_t*>(src) + lane);
    const float x0 = __uint_as_float(bits << 16), x1 = __uint_as_float(bits & 0xFFFF0000u);
    float a = fmaxf(fabsf(x0), fabsf(x1));
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) a = fmaxf(a, __shfl_xor_sync(0xffffffffu, a, o));
    uint32_t code = 0;
    float scale = 0.f;
    if (a > 0.f) {
      const float inv = __fdiv_rn(448.f, a);
      scale = __fdiv_rn(a, 448.f);
      code = e4m3x2(__fmul_rn(x0, inv), __fmul_rn(x1, inv));
    }
    if (which == 0) {
      reinterpret_cast<uint16_t*>(p.k8 + (blk * kPage + slot) * kHeadDim)[lane] = (uint16_t)code;
      if (lane == 0) p.k_scale[blk * kPage + slot] = scale;
    } else {
      uint8_t* col = p.v8 + blk * kF8Block + slot;  // transposed block: [dim][key]
      col[(2 * lane) * kPage] = (uint8_t)(code & 0xFF);
      col[(2 * lane + 1) * kPage] = (uint8_t)(code >> 8);
      if (lane == 0) p.v_scale[blk * kPage + slot] = scale;
    }
  }
}

// ------------------------------------------------------------------ launch

cudaError_t launch_kv_append_fp8(const void* k_new, const void* v_new, void* k8, void* v8, float* k_scale,
                                 float* v_scale, const int32_t* block_table, const int32_t* seq_lens,
                                 const int32_t* qsl, int32_t* status, int32_t num_seqs, int32_t total_q,
                                 int32_t max_pages, int32_t num_pages, int32_t num_kv_heads, cudaStream_t stream) {
  F8AppendParams p;
  p.k_new = static_cast<const __nv_bfloat16*>(k_new);
  p.v_new = static_cast<const __nv_bfloat16*>(v_new);
  p.k8 = static_cast<uint8_t*>(k8);
  p.v8 = static_cast<uint8_t*>(v8);
  p.k_scale = k_scale;
  p.v_scale = v_scale;
  p.block_table = block_table;
  p.seq_lens = seq_lens;
  p.qsl = qsl;
  p.status = status;
  p.num_seqs = num_seqs;
  p.total_q = total_q;
  p.max_pages = max_pages;
  p.num_pages = num_pages;
  p.num_kv_heads = num_kv_heads;
  const int64_t warps = (int64_t)total_q * num_kv_heads;
  const int grid = (int)((warps + kF8AppendWarps - 1) / kF8AppendWarps);
  kv_append_fp8_kernel<<<grid, kF8AppendWarps * 32, 0, stream>>>(p);
  return cudaGetLastError();
}

cudaError_t launch_decode_fp8(const void* k8, const void* v8, const float* k_scale, const float* v_scale,
                              const AttnParams& p, int grid, bool cascade, cudaStream_t stream) {
  F8Pools pools;
  pools.k8 = static_cast<const uint8_t*>(k8);
  pools.v8 = static_cast<const uint8_t*>(v8);
  pools.k_scale = k_scale;
  pools.v_scale = v_scale;
  if (cascade)
    decode_fp8_kernel<4><<<grid, kF8Warps * 32, decode_fp8_smem_bytes(), stream>>>(pools, p);
  else
    decode_fp8_kernel<1><<<grid, kF8Warps * 32, decode_fp8_smem_bytes(), stream>>>(pools, p);
  return cudaGetLastError();
}

cudaError_t prepare_fp8_kernels(int* blocks_per_sm_decode, int* blocks_per_sm_cascade) {
  cudaError_t e;
  e = cudaFuncSetAttribute(decode_fp8_kernel<1>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           (int)decode_fp8_smem_bytes());
  if (e != cudaSuccess) return e;
  e = cudaFuncSetAttribute(decode_fp8_kernel<4>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           (int)decode_fp8_smem_bytes());
  if (e != cudaSuccess) return e;
  e = cudaFuncSetAttribute(decode_fp8_kernel<1>, cudaFuncAttributePreferredSharedMemoryCarveout,
                           cudaSharedmemCarveoutMaxShared);
  if (e != cudaSuccess) return e;
  e = cudaFuncSetAttribute(decode_fp8_kernel<4>, cudaFuncAttributePreferredSharedMemoryCarveout,
                           cudaSharedmemCarveoutMaxShared);
  if (e != cudaSuccess) return e;
  e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(blocks_per_sm_decode, decode_fp8_kernel<1>, kF8Warps * 32,
                                                    decode_fp8_smem_bytes());
  if (e != cudaSuccess) return e;
  return cudaOccupancyMaxActiveBlocksPerMultiprocessor(blocks_per_sm_cascade, decode_fp8_kernel<4>, kF8Warps * 32,
                                                       decode_fp8_smem_bytes());
}

}  // namespace mcpu
