// fp8 (e4m3) KV pages: the quantizing KV append and the split-KV decode /
// cascade kernel that reads them (a storage variant; the paper keeps bf16).
//
// Storage: one 2176-byte block per (page, kv head), blocks ordered
// [page][kv head]:
//   bytes    0..1023  K codes [16 keys][64 dims] (row-major)
//   bytes 1024..2047  V codes in MMA-fragment order: for h in {0, 1}, lane
//                     (r, c) = (l / 4, l % 4) and j in 0..3, bytes
//                     1024 + 512 h + 16 l + 4 j + i hold dim
//                     d = 16 (2h + j / 2) + 8 (j % 2) + r of key 4c + i
//   bytes 2048..2175  scales: 16 bytes per r in 0..7 = K scale of keys
//                     a = 4(r / 2) + r % 2 and a + 2, then V scale of both
// so that one bulk copy brings a page and every operand of a lane is one
// 128-bit shared-memory load (two for K, two for V, one for the scales).
// Each new row x (64 bf16 values) is stored as a = max|x_i|, scale = a / 448
// and code_i = e4m3(x_i * (448 / a)) (round to nearest even, saturating), in
// float arithmetic; an all-zero row stores zeros. A key is code * scale.
//
// Decode over fp8 pages follows the bf16 kernel (one warp per work item, a
// per-warp ring of pages filled by one bulk copy each, m16n8k16 tensor-core
// tiles, online softmax in fp32, partials merged by log-sum-exp):
//   - codes become fp16 MMA operands by the hardware conversion of code
//     pairs (exact: every e4m3 value is an fp16 value);
//   - S = K q: q (bf16) enters as fp16 times a power of two per query
//     vector (largest entry in [2^14, 2^15), exact for every bf16 entry
//     above 2^-28 of it); each score is then scaled by its key's scale, the
//     power of two and the softmax scale;
//   - O += P' V: P' = p * v_scale * 2^F in fp16, F a per-item power of two
//     that only decreases so that v_scale * 2^F < 1 and P' < 2^8; the
//     accumulator is rescaled when F drops and divided by 2^F at the end.
// MMA row r of the score tile is key 4(r/2) + (r%2) and row r + 8 is that
// key + 2, so that movmatrix turns the score fragment into the P' operand
// whose k-slots 2c, 2c + 1, 2c + 8, 2c + 9 are keys 4c .. 4c + 3, the keys
// of one 32-bit word of V codes. The running max is lazy: scores are
// exponentiated against a reference that is only raised (with the rescale)
// when a score exceeds it by more than 8 (p <= 2^8), and F is only lowered
// when a page's V scale needs it; both checks are one warp vote per page.
// On pages that a row sees only in part (its first and last), codes of
// invisible V slots are zeroed before conversion (unwritten slots may hold
// any byte, e4m3 NaN included) and their scores masked; a page outside the
// pool is skipped.
#include <cuda_fp16.h>

#include "common.cuh"

namespace mcpu {

constexpr int kF8Warps = 4;
constexpr int kF8Stages = 6;
constexpr int kF8Codes = kPage * kHeadDim;  // 1024 codes per (page, kv head) for K, and for V
constexpr int kF8VOff = kF8Codes;
constexpr int kF8ScaleOff = 2 * kF8Codes;
constexpr int kF8BlockBytes = 2 * kF8Codes + 2 * kPage * 4;  // 2176
constexpr float kF8Lazy = 8.f;      // scores may exceed the reference max by this much (base 2)
constexpr float kF8NoMax = -1e30f;  // reference max before the first visible key
constexpr int kF8RingBytes = kF8Stages * kF8BlockBytes;

size_t decode_fp8_smem_bytes() {
  return 128 /* alignment slack */ + (size_t)kF8Warps * kF8RingBytes + (size_t)kF8Warps * kF8Stages * 8;
}

// e4m3 codes of x0 (low byte) and x1 (high byte): nearest, ties to even,
// saturating at +-448.
__device__ __forceinline__ uint32_t e4m3x2(float x0, float x1) {
  uint16_t d;
  asm("cvt.rn.satfinite.e4m3x2.f32 %0, %1, %2;" : "=h"(d) : "f"(x1), "f"(x0));
  return d;
}
__device__ __forceinline__ uint32_t pack_f16x2(float lo, float hi) {
  __half2 v = __floats2half2_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}
// the four codes of a word as two exact f16 pairs: (bytes 0, 1) and (2, 3)
__device__ __forceinline__ void f16x2x2_from_e4m3x4(uint32_t w, uint32_t& lo, uint32_t& hi) {
  asm("{\n\t.reg .b16 l16, h16;\n\t"
      "mov.b32 {l16, h16}, %2;\n\t"
      "cvt.rn.f16x2.e4m3x2 %0, l16;\n\t"
      "cvt.rn.f16x2.e4m3x2 %1, h16;\n\t}"
      : "=r"(lo), "=r"(hi)
      : "r"(w));
}

// 2^e as a float for -126 <= e <= 127
__device__ __forceinline__ float exp2i(int e) { return __uint_as_float((uint32_t)(e + 127) << 23); }

// floor(log2(x)) of a positive finite float (subnormals give -127)
__device__ __forceinline__ int ilog2f(float x) { return (int)((__float_as_uint(x) >> 23) & 0xFF) - 127; }

// Byte mask of the keys 4c..4c+3 of a page that lie in [lo, hi).
__device__ __forceinline__ uint32_t key_byte_mask(int c, int lo, int hi) {
  uint32_t m = 0;
#pragma unroll
  for (int i = 0; i < 4; ++i) m |= (4 * c + i >= lo && 4 * c + i < hi) ? (0xFFu << (8 * i)) : 0u;
  return m;
}

template <int NT>
__global__ void __launch_bounds__(kF8Warps * 32, NT == 1 ? 4 : 1)
    decode_fp8_kernel(const uint8_t* __restrict__ kv8, const AttnParams p) {
  // The cascade pass (NT > 1) may be launched programmatically after the
  // decode kernel: it waits for that kernel before it exits (see decode.cu).
  if ((NT == 1 ? header(p)->n_decode : header(p)->n_cascade) == 0) {  // nothing of this kind
    if (NT > 1) grid_dep_wait();
    return;
  }
  extern __shared__ uint8_t smem_raw[];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int r = lane >> 2, c = lane & 3;
  const int key_a = 4 * (r >> 1) + (r & 1), key_b = key_a + 2;  // keys of M rows r and r + 8
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
    // 16c .. 16c + 15 as fp16 of q * 2^eq; MMA step kk takes dims
    // 16c + 4kk, +1 (k-slots 2c, 2c + 1) and 16c + 4kk + 2, +3 (2c + 8, 2c + 9).
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
#pragma unroll
      for (int kk = 0; kk < 4; ++kk) {
        qb[nt][kk][0] = pack_f16x2(x[4 * kk] * up, x[4 * kk + 1] * up);
        qb[nt][kk][1] = pack_f16x2(x[4 * kk + 2] * up, x[4 * kk + 3] * up);
      }
      const float my_qm = exp2i(-eq) * p.scale_log2;
      qm[nt][0] = __shfl_sync(0xffffffffu, my_qm, (2 * c) * 4);
      qm[nt][1] = __shfl_sync(0xffffffffu, my_qm, (2 * c + 1) * 4);
    }

    // Page ids: lane i caches the id of page (chunk + i); lane 0 issues.
    const int n = pe - pb;
    int chunk_base = -32, pid_reg = 0;
    uint32_t bad_stages = 0;  // stages holding no page (warp-uniform)
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
    auto issue = [&](int k, uint32_t s) {  // page k of the item into ring stage s
      const int pid = page_id(k);
      bad_stages = pid < 0 ? (bad_stages | (1u << s)) : (bad_stages & ~(1u << s));
      if (lane == 0) {
        const uint32_t bar = bars + 8 * s;
        if (pid < 0) {
          mbar_arrive(bar);  // nothing to copy: the page is skipped
        } else {
          mbar_arrive_expect_tx(bar, kF8BlockBytes);
          bulk_load(ring + s * kF8BlockBytes, kv8 + ((size_t)pid * Hkv + kvh) * kF8BlockBytes, kF8BlockBytes, bar,
                    pol);
        }
      }
    };
    const int pre = n < kF8Stages ? n : kF8Stages;
    for (int k = 0; k < pre; ++k) issue(k, (seq + k) % kF8Stages);

    float m_ref[NT][2], l_run[NT][2], acc[4][NT][4];
#pragma unroll
    for (int nt = 0; nt < NT; ++nt) {
      m_ref[nt][0] = m_ref[nt][1] = kF8NoMax;
      l_run[nt][0] = l_run[nt][1] = 0.f;
#pragma unroll
      for (int mt = 0; mt < 4; ++mt)
#pragma unroll
        for (int e = 0; e < 4; ++e) acc[mt][nt][e] = 0.f;
    }
    int F = 125;           // P' = p * v_scale * 2^F; acc is held in units of 2^F
    float u_lim = 0.f;     // 2^-F: a V scale at or above it needs a lower F
    float pf = exp2i(F);

    bool timed_out = false;
    uint32_t s = seq % kF8Stages, phase = (seq / kF8Stages) & 1u;
    for (int k = 0; k < n; ++k) {
      const bool ok = __any_sync(0xffffffffu, mbar_wait(bars + 8 * s, phase));
      if (!ok) {
        timed_out = true;
        break;
      }
      if (!((bad_stages >> s) & 1u)) {
        const uint8_t* st = ring_ptr + s * kF8BlockBytes;
        const uint4 KA = *reinterpret_cast<const uint4*>(st + key_a * kHeadDim + 16 * c);
        const uint4 KB = *reinterpret_cast<const uint4*>(st + key_b * kHeadDim + 16 * c);
        const float4 sc = *reinterpret_cast<const float4*>(st + kF8ScaleOff + 16 * r);  // ks_a, ks_b, vs_a, vs_b
        const uint4 V0 = *reinterpret_cast<const uint4*>(st + kF8VOff + 16 * lane);
        const uint4 V1 = *reinterpret_cast<const uint4*>(st + kF8VOff + 512 + 16 * lane);

        // S^T[16 keys x 8*NT query vectors] in units of q * 2^eq * K codes
        float cc[NT][4];
#pragma unroll
        for (int nt = 0; nt < NT; ++nt) cc[nt][0] = cc[nt][1] = cc[nt][2] = cc[nt][3] = 0.f;
        {
          const uint32_t wa[4] = {KA.x, KA.y, KA.z, KA.w}, wb[4] = {KB.x, KB.y, KB.z, KB.w};
#pragma unroll
          for (int kk = 0; kk < 4; ++kk) {
            uint32_t a0, a1, a2, a3;
            f16x2x2_from_e4m3x4(wa[kk], a0, a2);
            f16x2x2_from_e4m3x4(wb[kk], a1, a3);
#pragma unroll
            for (int nt = 0; nt < NT; ++nt) mma_f16_16816(cc[nt], a0, a1, a2, a3, qb[nt][kk][0], qb[nt][kk][1]);
          }
        }

        // t = score - reference (base 2): one FFMA per score
        float fk[NT][4], tv[NT][4];
#pragma unroll
        for (int nt = 0; nt < NT; ++nt) {
          fk[nt][0] = sc.x * qm[nt][0];
          fk[nt][1] = sc.x * qm[nt][1];
          fk[nt][2] = sc.y * qm[nt][0];
          fk[nt][3] = sc.y * qm[nt][1];
#pragma unroll
          for (int i = 0; i < 4; ++i) tv[nt][i] = fmaf(cc[nt][i], fk[nt][i], -m_ref[nt][i & 1]);
        }
        float u0 = sc.z, u1 = sc.w;
        bool v0 = true, v1 = true;
        uint32_t vw[8] = {V0.x, V0.y, V0.z, V0.w, V1.x, V1.y, V1.z, V1.w};
        // a row's first and last pages may hold keys it does not see
        const int pk = (pb + k) * kPage;
        if (NT == 1 && (pk < first_key || pk + kPage > seq_len)) {
          const int klo = max(first_key - pk, 0), khi = min(seq_len - pk, kPage);
          v0 = key_a >= klo && key_a < khi;
          v1 = key_b >= klo && key_b < khi;
#pragma unroll
          for (int nt = 0; nt < NT; ++nt) {
            tv[nt][0] = v0 ? tv[nt][0] : -INFINITY;
            tv[nt][1] = v0 ? tv[nt][1] : -INFINITY;
            tv[nt][2] = v1 ? tv[nt][2] : -INFINITY;
            tv[nt][3] = v1 ? tv[nt][3] : -INFINITY;
          }
          u0 = v0 ? u0 : 0.f;
          u1 = v1 ? u1 : 0.f;
          const uint32_t vmask = key_byte_mask(c, klo, khi);
#pragma unroll
          for (int i = 0; i < 8; ++i) vw[i] &= vmask;
        }

        // rare: a score above the reference by more than kF8Lazy, or a V
        // scale that needs a lower F
        bool over = fmaxf(u0, u1) >= u_lim;
#pragma unroll
        for (int nt = 0; nt < NT; ++nt)
          over |= fmaxf(fmaxf(tv[nt][0], tv[nt][2]), fmaxf(tv[nt][1], tv[nt][3])) > kF8Lazy;
        if (__any_sync(0xffffffffu, over)) {
          float um = fmaxf(u0, u1);
          um = fmaxf(um, __shfl_xor_sync(0xffffffffu, um, 4));
          um = fmaxf(um, __shfl_xor_sync(0xffffffffu, um, 8));
          um = fmaxf(um, __shfl_xor_sync(0xffffffffu, um, 16));
          int F_new = F;
          if (um >= u_lim && um > 0.f) F_new = max(min(F, -1 - ilog2f(um)), -125);
          const float dF = F_new - F >= -126 ? exp2i(F_new - F) : 0.f;
          F = F_new;
          pf = exp2i(F);
          u_lim = exp2i(-F);
#pragma unroll
          for (int nt = 0; nt < NT; ++nt) {
            // exact scores again (the reference may still be the initial -1e30)
            float sx[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) sx[i] = ((i < 2) ? v0 : v1) ? cc[nt][i] * fk[nt][i] : -INFINITY;
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
            const float ac0 = al0 * dF, ac1 = al1 * dF;
#pragma unroll
            for (int mt = 0; mt < 4; ++mt) {
              acc[mt][nt][0] *= ac0;
              acc[mt][nt][1] *= ac1;
              acc[mt][nt][2] *= ac0;
              acc[mt][nt][3] *= ac1;
            }
          }
        }
        const float w0 = u0 * pf, w1 = u1 * pf;

        uint32_t pb0[NT], pb1[NT];
#pragma unroll
        for (int nt = 0; nt < NT; ++nt) {
          const float p00 = ex2_approx(tv[nt][0]), p01 = ex2_approx(tv[nt][1]);
          const float p10 = ex2_approx(tv[nt][2]), p11 = ex2_approx(tv[nt][3]);
          l_run[nt][0] += p00 + p10;
          l_run[nt][1] += p01 + p11;
          pb0[nt] = movmatrix_trans(pack_f16x2(p00 * w0, p01 * w0));  // keys 4c, 4c + 1 of column r
          pb1[nt] = movmatrix_trans(pack_f16x2(p10 * w1, p11 * w1));  // keys 4c + 2, 4c + 3
        }

        // O^T[64 dims x 8*NT] += V^T P'^T over dims 16 mt + r and 16 mt + 8 + r
#pragma unroll
        for (int mt = 0; mt < 4; ++mt) {
          uint32_t a0, a1, a2, a3;
          f16x2x2_from_e4m3x4(vw[2 * mt], a0, a2);
          f16x2x2_from_e4m3x4(vw[2 * mt + 1], a1, a3);
#pragma unroll
          for (int nt = 0; nt < NT; ++nt) mma_f16_16816(acc[mt][nt], a0, a1, a2, a3, pb0[nt], pb1[nt]);
        }
      }

      // release the stage to the async proxy, then refill it
      fence_proxy_async();
      __syncwarp();
      if (k + kF8Stages < n) issue(k + kF8Stages, s);
      if (++s == kF8Stages) {
        s = 0;
        phase ^= 1u;
      }
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
    const float unit = exp2i(-F);  // acc -> output units (|F| <= 125)
    constexpr int kLd = kHeadDim + 4;    // padded rows: conflict-free stores, 16-byte aligned rows
    float* so = scratch;                 // [8*NT][kLd]
    float* sl = scratch + 8 * NT * kLd;  // [8*NT] base-2 lse
#pragma unroll
    for (int nt = 0; nt < NT; ++nt) {
#pragma unroll
      for (int e = 0; e < 2; ++e) {
        const int qv = nt * 8 + 2 * c + e;
        const float l = l_run[nt][e];
        const float m = l > 0.f ? m_ref[nt][e] : -INFINITY;
        float inv = l > 0.f ? 1.f / l : 0.f;
        float lse2 = l > 0.f ? m + __log2f(l) : -INFINITY;
        if (NT == 1 && p.sinks != nullptr && slot < 0 && qv < g)
          inv = finish_with_sink(m, l, sink_log2(p, kvh * g + qv), &lse2);
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
      const float2 o = *reinterpret_cast<const float2*>(so + qv * kLd + 2 * lane);
      const float o0 = o.x, o1 = o.y;
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
  // no item left for this warp: the grid after this one may launch
  grid_dep_launch();
  if (NT > 1) grid_dep_wait();
}

// ------------------------------------------------------------ fp8 KV append

constexpr int kF8AppendWarps = 8;

struct F8AppendParams {
  const __nv_bfloat16* k_new;  // [T, Hkv, D]
  const __nv_bfloat16* v_new;
  uint8_t* kv8;                // [P, Hkv] blocks of kF8BlockBytes
  const int32_t* block_table;
  const int32_t* seq_lens;
  const int32_t* qsl;
  int32_t* status;
  int32_t num_seqs, total_q, max_pages, num_pages, num_kv_heads;
};

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
  uint8_t* blk = p.kv8 + ((size_t)page * p.num_kv_heads + h) * kF8BlockBytes;
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
    // scale slot of this key: r = 2 (slot / 4) + slot % 2, the key's half (slot / 2) % 2
    const int sc_idx = 4 * (2 * (slot >> 2) + (slot & 1)) + ((slot >> 1) & 1);
    if (which == 0) {
      reinterpret_cast<uint16_t*>(blk + slot * kHeadDim)[lane] = (uint16_t)code;
      if (lane == 0) reinterpret_cast<float*>(blk + kF8ScaleOff)[sc_idx] = scale;
    } else {
#pragma unroll
      for (int e = 0; e < 2; ++e) {  // dim d = 2 lane + e in fragment order
        const int d = 2 * lane + e, mt = d >> 4, hf = (d >> 3) & 1, rr = d & 7;
        const int off = kF8VOff + (mt >> 1) * 512 + (4 * rr + (slot >> 2)) * 16 + 4 * ((mt & 1) * 2 + hf) + (slot & 3);
        blk[off] = (uint8_t)(e ? code >> 8 : code & 0xFF);
      }
      if (lane == 0) reinterpret_cast<float*>(blk + kF8ScaleOff)[sc_idx + 2] = scale;
    }
  }
}

// ------------------------------------------------------------------ launch

cudaError_t launch_kv_append_fp8(const void* k_new, const void* v_new, void* kv8, const int32_t* block_table,
                                 const int32_t* seq_lens, const int32_t* qsl, int32_t* status, int32_t num_seqs,
                                 int32_t total_q, int32_t max_pages, int32_t num_pages, int32_t num_kv_heads,
                                 cudaStream_t stream) {
  F8AppendParams p;
  p.k_new = static_cast<const __nv_bfloat16*>(k_new);
  p.v_new = static_cast<const __nv_bfloat16*>(v_new);
  p.kv8 = static_cast<uint8_t*>(kv8);
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

// `programmatic` (cascade pass only): launched with programmatic stream
// serialization right after the decode kernel on the same stream.
cudaError_t launch_decode_fp8(const void* kv8, const AttnParams& p, int grid, bool cascade, cudaStream_t stream,
                              bool programmatic) {
  const uint8_t* pool = static_cast<const uint8_t*>(kv8);
  LaunchCfg lc(dim3(grid), dim3(kF8Warps * 32), decode_fp8_smem_bytes(), stream, programmatic && cascade);
  return cascade ? cudaLaunchKernelEx(&lc.cfg, decode_fp8_kernel<4>, pool, p)
                 : cudaLaunchKernelEx(&lc.cfg, decode_fp8_kernel<1>, pool, p);
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
