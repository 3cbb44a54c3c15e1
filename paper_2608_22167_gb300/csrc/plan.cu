// Work planner: one CTA reads seq_lens / query_start_loc / block_table on the
// device and writes the work lists of the attention kernels into the
// workspace, so a forward call needs no host round trip and can be captured
// in a CUDA graph.
//
// It decides, per row: decode (L = 1), append (L > 1) or nothing; for decode
// rows, the KV split length and the partial-result slots merged later by
// log-sum-exp; for runs of adjacent rows whose block tables begin with the
// same physical pages (the G samples of a GRPO task sharing their prompt,
// paper §4), the shared prefix that one cascade pass reads once for the
// whole group; for append rows, the query tiles of the chunk kernel.
#include "common.cuh"

namespace mcpu {

namespace {

constexpr int kWarps = kPlanThreads / 32;
constexpr int R = kRowsPerPlanThread;  // rows owned by each thread: tid * R + i

struct ScanBuf {
  int warp[kWarps + 1];
};

// Exclusive prefix sum over the whole CTA of one value per thread; the CTA
// total is returned through *total. Every thread must call it.
__device__ int cta_scan(int v, int* total, ScanBuf& sb) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  int x = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    int y = __shfl_up_sync(0xffffffffu, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) sb.warp[warp] = x;
  __syncthreads();
  if (warp == 0) {
    int s = sb.warp[lane];
    int t = s;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      int y = __shfl_up_sync(0xffffffffu, t, o);
      if (lane >= o) t += y;
    }
    sb.warp[lane] = t - s;
    if (lane == 31) sb.warp[kWarps] = t;
  }
  __syncthreads();
  const int res = sb.warp[warp] + x - v;
  *total = sb.warp[kWarps];
  __syncthreads();
  return res;
}

// Exclusive scan of R values per thread (rows tid*R .. tid*R+R-1).
__device__ void cta_scan_rows(const int (&v)[R], int (&out)[R], int* total, ScanBuf& sb) {
  int s = 0;
#pragma unroll
  for (int i = 0; i < R; ++i) s += v[i];
  int base = cta_scan(s, total, sb);
#pragma unroll
  for (int i = 0; i < R; ++i) {
    out[i] = base;
    base += v[i];
  }
}

__device__ __forceinline__ int cdiv(int a, int b) { return (a + b - 1) / b; }

}  // namespace

// Dynamic shared memory: per-row arrays (kMaxSeqs entries each).
struct PlanSmem {
  int S[kMaxSeqs];
  int lcp[kMaxSeqs];
  int gid[kMaxSeqs];
  int grp_pages[kMaxSeqs];   // shared full pages of a group (min over the run)
  int grp_ndec[kMaxSeqs];    // decode rows in the group
  int grp_base[kMaxSeqs];    // smallest member rank in the group
  signed char kind[kMaxSeqs];  // 0 none / invalid, 1 decode, 2 append
  ScanBuf sb;
  int bad_global;
};

__global__ void __launch_bounds__(kPlanThreads, 1) plan_kernel(AttnParams p) {
  extern __shared__ __align__(16) uint8_t plan_smem_raw[];
  PlanSmem& sm = *reinterpret_cast<PlanSmem*>(plan_smem_raw);
  PlanHeader* hdr = header(p);
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int B = p.num_seqs;
  const int Hkv = p.num_kv_heads;
  const int tile_tok = kAppendRows / p.group;
  const int sub_cap = 32 / p.group;  // query vectors of a cascade item: 32

  if (tid == 0) {
    int bad = (p.qsl[0] != 0 || p.qsl[B] != p.total_q) ? 1 : 0;
    sm.bad_global = bad;
    if (bad) atomicOr(&hdr->status, kStatusBadLengths);
  }
  __syncthreads();
  if (sm.bad_global) {
    if (tid == 0) {
      hdr->n_decode = hdr->n_cascade = hdr->n_append = hdr->n_merge = 0;
      hdr->n_parts = 0;
      hdr->append_ticket = 0;
    }
    return;
  }

  // ---- phase 1: per-row kind and lengths
  int S[R], L[R], Q0[R], kind[R];
#pragma unroll
  for (int i = 0; i < R; ++i) {
    const int r = tid * R + i;
    S[i] = L[i] = Q0[i] = kind[i] = 0;
    if (r < B) {
      const int q0 = p.qsl[r], q1 = p.qsl[r + 1];
      const int len = q1 - q0, s = p.seq_lens[r];
      const bool bad = len < 0 || s < len || s > p.max_pages * kPage;
      if (bad) {
        atomicOr(&hdr->status, kStatusBadLengths);
      } else {
        S[i] = s;
        L[i] = len;
        Q0[i] = q0;
        kind[i] = len == 0 ? 0 : (len == 1 ? 1 : 2);
      }
      sm.S[r] = bad ? -1 : s;
      sm.kind[r] = (signed char)kind[i];
      sm.lcp[r] = 0;
      sm.grp_pages[r] = 0x7fffffff;
      sm.grp_ndec[r] = 0;
      sm.grp_base[r] = 0x7fffffff;
    }
  }
  __syncthreads();

  // ---- phase 2: shared-prefix groups (full-context calls only)
  const bool cascade = p.cascade_enabled && p.window <= 0;
  if (cascade) {
    for (int r = warp + 1; r < B; r += kWarps) {
      const int sa = sm.S[r - 1], sb = sm.S[r];
      if (sa < 0 || sb < 0) continue;
      const int lim = min(sa, sb) / kPage;  // pages full in both rows
      const int* ba = p.block_table + (size_t)(r - 1) * p.max_pages;
      const int* bb = p.block_table + (size_t)r * p.max_pages;
      int n = 0;
      for (int base = 0; base < lim; base += 32) {
        const int i = base + lane;
        const bool eq = i < lim && __ldg(ba + i) == __ldg(bb + i);
        const unsigned m = __ballot_sync(0xffffffffu, eq);
        if (m == 0xffffffffu) {
          n += 32;
          continue;
        }
        n += __ffs(~m) - 1;
        break;
      }
      if (lane == 0) sm.lcp[r] = min(n, lim);
    }
  }
  __syncthreads();

  // group id = (number of run starts up to and including r) - 1
  {
    int st[R], ex[R], tot;
#pragma unroll
    for (int i = 0; i < R; ++i) {
      const int r = tid * R + i;
      st[i] = (r < B && (r == 0 || !cascade || sm.lcp[r] < kMinSharedPages)) ? 1 : 0;
    }
    cta_scan_rows(st, ex, &tot, sm.sb);
#pragma unroll
    for (int i = 0; i < R; ++i) {
      const int r = tid * R + i;
      if (r < B) sm.gid[r] = ex[i] + st[i] - 1;
    }
  }
  __syncthreads();
  if (cascade) {
#pragma unroll
    for (int i = 0; i < R; ++i) {
      const int r = tid * R + i;
      if (r >= B) continue;
      const int g = sm.gid[r];
      if (r > 0 && sm.gid[r - 1] == g) atomicMin(&sm.grp_pages[g], sm.lcp[r]);
      if (kind[i] == 1) {
        atomicMin(&sm.grp_pages[g], S[i] / kPage);
        atomicAdd(&sm.grp_ndec[g], 1);
      }
    }
  }
  __syncthreads();

  // members: decode rows of a group with >= 2 decode rows and a long enough prefix
  int member[R], mrank[R], n_members_total;
  {
#pragma unroll
    for (int i = 0; i < R; ++i) {
      const int r = tid * R + i;
      member[i] = 0;
      if (cascade && r < B && kind[i] == 1) {
        const int g = sm.gid[r];
        member[i] = (sm.grp_ndec[g] >= 2 && sm.grp_pages[g] >= kMinSharedPages) ? 1 : 0;
      }
    }
    cta_scan_rows(member, mrank, &n_members_total, sm.sb);
#pragma unroll
    for (int i = 0; i < R; ++i)
      if (member[i]) atomicMin(&sm.grp_base[sm.gid[tid * R + i]], mrank[i]);
  }
  __syncthreads();

  // ---- phase 3: split length
  int own_pb[R], own_pe[R], gpages[R], nsub[R], sub_idx[R], sub_first[R];
  int w_m = 0, w_lb = 0;
#pragma unroll
  for (int i = 0; i < R; ++i) {
    const int r = tid * R + i;
    own_pb[i] = own_pe[i] = gpages[i] = nsub[i] = sub_idx[i] = sub_first[i] = 0;
    if (r >= B || kind[i] != 1) continue;
    const int first_key = p.window > 0 ? max(0, S[i] - p.window) : 0;
    own_pe[i] = cdiv(S[i], kPage);
    own_pb[i] = first_key / kPage;
    if (member[i]) {
      const int g = sm.gid[r];
      const int nd = sm.grp_ndec[g];
      gpages[i] = sm.grp_pages[g];
      own_pb[i] = gpages[i];
      nsub[i] = cdiv(nd, sub_cap);
      const int idx = mrank[i] - sm.grp_base[g];
      sub_idx[i] = idx * nsub[i] / nd;
      // first member index of this subgroup: ceil(sub * nd / nsub)
      sub_first[i] = (idx == cdiv(sub_idx[i] * nd, nsub[i])) ? 1 : 0;
    }
    const int own = own_pe[i] - own_pb[i];
    w_m += own + (member[i] ? gpages[i] : 0);
    w_lb += own + (sub_first[i] ? gpages[i] : 0);
  }
  int tot_wm, tot_wlb;
  cta_scan(w_m, &tot_wm, sm.sb);
  cta_scan(w_lb, &tot_wlb, sm.sb);
  const int c_bound = max(1, cdiv(tot_wm, kSplitBudget));
  int C;
  if (p.forced_split_pages > 0) {
    C = max(p.forced_split_pages, c_bound);
  } else {
    const long long denom = 4LL * max(p.total_warps_hint, 1);
    const int c_lb = (int)((((long long)tot_wlb) * Hkv + denom - 1) / denom);
    C = max(kMinSplitPages, max(c_lb, c_bound));
  }

  // ---- phase 4: decode items, partial slots, merge rows
  int n_own[R], n_cs[R], parts[R], direct[R];
#pragma unroll
  for (int i = 0; i < R; ++i) {
    n_own[i] = (kind[i] == 1) ? cdiv(own_pe[i] - own_pb[i], C) : 0;
    n_cs[i] = member[i] ? cdiv(gpages[i], C) : 0;
    parts[i] = n_own[i] + n_cs[i];
    direct[i] = (kind[i] == 1 && !member[i] && parts[i] == 1) ? 1 : 0;
  }
  int pc[R], part_off[R], item_off[R], is_merge[R], merge_off[R];
  int tot_parts, tot_items, tot_merge;
#pragma unroll
  for (int i = 0; i < R; ++i) {
    pc[i] = (kind[i] == 1 && !direct[i]) ? parts[i] : 0;
    is_merge[i] = pc[i] > 0 ? 1 : 0;
  }
  cta_scan_rows(pc, part_off, &tot_parts, sm.sb);
  cta_scan_rows(n_own, item_off, &tot_items, sm.sb);
  cta_scan_rows(is_merge, merge_off, &tot_merge, sm.sb);

  // ---- phase 5: cascade subgroups (one record per split of each subgroup)
  int sg_splits[R], sg_off[R], tot_cascade;
#pragma unroll
  for (int i = 0; i < R; ++i) sg_splits[i] = sub_first[i] ? n_cs[i] : 0;
  cta_scan_rows(sg_splits, sg_off, &tot_cascade, sm.sb);

  // ---- phase 6: append tiles
  int tiles[R], tile_off[R], tot_tiles;
#pragma unroll
  for (int i = 0; i < R; ++i) tiles[i] = kind[i] == 2 ? cdiv(L[i], tile_tok) : 0;
  cta_scan_rows(tiles, tile_off, &tot_tiles, sm.sb);

  const bool overflow = tot_items > p.lay.max_decode || tot_cascade > p.lay.max_cascade ||
                        tot_tiles > p.lay.max_append || tot_parts > p.lay.max_parts;
  if (overflow) {
    if (tid == 0) {
      atomicOr(&hdr->status, kStatusPlanOverflow);
      hdr->n_decode = hdr->n_cascade = hdr->n_append = hdr->n_merge = 0;
      hdr->n_parts = 0;
      hdr->append_ticket = 0;
    }
    return;
  }

  DecodeItem* ditems = reinterpret_cast<DecodeItem*>(p.ws + p.lay.decode_items);
  CascadeItem* citems = reinterpret_cast<CascadeItem*>(p.ws + p.lay.cascade_items);
  CascadeMember* members = reinterpret_cast<CascadeMember*>(p.ws + p.lay.members);
  AppendItem* aitems = reinterpret_cast<AppendItem*>(p.ws + p.lay.append_items);
  MergeRow* mrows = reinterpret_cast<MergeRow*>(p.ws + p.lay.merge_rows);

#pragma unroll
  for (int i = 0; i < R; ++i) {
    const int r = tid * R + i;
    if (r >= B) continue;
    if (kind[i] == 1) {
      const int first_key = p.window > 0 ? max(0, S[i] - p.window) : 0;
      for (int k = 0; k < n_own[i]; ++k) {
        DecodeItem it;
        it.row = r;
        it.token = Q0[i];
        it.seq_len = S[i];
        it.first_key = first_key;
        it.page_begin = own_pb[i] + k * C;
        it.page_end = min(own_pe[i], own_pb[i] + (k + 1) * C);
        it.slot = direct[i] ? -1 : part_off[i] + n_cs[i] + k;
        it.pad = 0;
        ditems[item_off[i] + k] = it;
      }
      if (is_merge[i]) {
        MergeRow m;
        m.token = Q0[i];
        m.n_parts = parts[i];
        m.part_off = part_off[i];
        m.pad = 0;
        mrows[merge_off[i]] = m;
      }
      if (member[i]) {
        CascadeMember cm;
        cm.row = r;
        cm.token = Q0[i];
        cm.part_off = part_off[i];
        cm.pad = 0;
        members[mrank[i]] = cm;
      }
      if (sub_first[i]) {
        const int g = sm.gid[r];
        const int nd = sm.grp_ndec[g];
        const int first = cdiv(sub_idx[i] * nd, nsub[i]);
        const int next = cdiv((sub_idx[i] + 1) * nd, nsub[i]);
        for (int k = 0; k < n_cs[i]; ++k) {
          CascadeItem c;
          c.member_off = sm.grp_base[g] + first;
          c.n_members = next - first;
          c.page_begin = k * C;
          c.page_end = min(gpages[i], (k + 1) * C);
          c.split = k;
          c.first_row = r;
          c.pad0 = c.pad1 = 0;
          citems[sg_off[i] + k] = c;
        }
      }
    } else if (kind[i] == 2) {
      for (int k = 0; k < tiles[i]; ++k) {
        AppendItem a;
        a.row = r;
        a.token_begin = Q0[i] + k * tile_tok;
        a.n_tok = min(tile_tok, L[i] - k * tile_tok);
        a.seq_len = S[i];
        a.pos_begin = S[i] - L[i] + k * tile_tok;
        a.key_begin = p.window > 0 ? max(0, a.pos_begin - p.window + 1) : 0;
        a.key_end = a.pos_begin + a.n_tok;
        a.pad = 0;
        aitems[tile_off[i] + k] = a;
      }
    }
  }
  if (tid == 0) {
    hdr->n_decode = tot_items;
    hdr->n_cascade = tot_cascade;
    hdr->n_append = tot_tiles;
    hdr->n_merge = tot_merge;
    hdr->split_pages = C;
    hdr->n_parts = tot_parts;
    hdr->append_ticket = 0;
  }
}

size_t plan_smem_bytes() { return sizeof(PlanSmem); }

cudaError_t launch_plan(const AttnParams& p, cudaStream_t stream) {
  static_assert(sizeof(PlanSmem) < 200 * 1024, "planner shared memory");
  plan_kernel<<<1, kPlanThreads, sizeof(PlanSmem), stream>>>(p);
  return cudaGetLastError();
}

cudaError_t prepare_plan_kernel() {
  return cudaFuncSetAttribute(plan_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sizeof(PlanSmem));
}

}  // namespace mcpu
