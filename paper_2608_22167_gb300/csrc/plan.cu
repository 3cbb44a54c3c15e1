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
//
// Per-row quantities are held in shared memory; every count becomes an
// offset by a CTA-wide prefix sum, and the records are then written by all
// threads in parallel (each finds its row by binary search over the offsets).
#include "common.cuh"

namespace mcpu {

namespace {

// The planner runs as one CTA of NT threads (256 for up to 512 rows, else
// 1024), each owning R = 2 consecutive rows for the scans.
constexpr int R = kRowsPerPlanThread;  // rows owned by each thread: tid * R + i

struct ScanBuf {
  int warp[kPlanThreads / 32 + 1];
};

// Exclusive prefix sum over the whole CTA of one value per thread; the CTA
// total is returned through *total. Every thread must call it.
template <int NT>
__device__ int cta_scan(int v, int* total, ScanBuf& sb) {
  constexpr int kWarps = NT / 32;
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
    const int s = lane < kWarps ? sb.warp[lane] : 0;
    int t = s;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      int y = __shfl_up_sync(0xffffffffu, t, o);
      if (lane >= o) t += y;
    }
    if (lane < kWarps) sb.warp[lane] = t - s;
    if (lane == kWarps - 1) sb.warp[kWarps] = t;
  }
  __syncthreads();
  const int res = sb.warp[warp] + x - v;
  *total = sb.warp[kWarps];
  __syncthreads();
  return res;
}

// Exclusive scan of a per-row array in shared memory (rows tid*R .. +R-1),
// written back in place; returns the total.
template <int NT>
__device__ int scan_rows(int* a, int B, ScanBuf& sb) {
  int v[R], s = 0;
#pragma unroll
  for (int i = 0; i < R; ++i) {
    const int r = threadIdx.x * R + i;
    v[i] = r < B ? a[r] : 0;
    s += v[i];
  }
  int total;
  int base = cta_scan<NT>(s, &total, sb);
#pragma unroll
  for (int i = 0; i < R; ++i) {
    const int r = threadIdx.x * R + i;
    if (r < B) a[r] = base;
    base += v[i];
  }
  __syncthreads();
  return total;
}

// Last row r with off[r] <= e (rows with no records share the next row's
// offset, so the last one is always a row that owns record e).
__device__ __forceinline__ int owner_row(const int* off, int B, int e) {
  int lo = 0, hi = B;  // off[lo] <= e < off[hi] (off[B] = +inf)
  while (hi - lo > 1) {
    const int mid = (lo + hi) >> 1;
    if (off[mid] <= e) lo = mid; else hi = mid;
  }
  return lo;
}

__device__ __forceinline__ int cdiv(int a, int b) { return (a + b - 1) / b; }

}  // namespace

// Row flags
constexpr int kFlagMember = 1;    // decode row served by a cascade pass
constexpr int kFlagDirect = 2;    // decode row with one part: writes out/lse itself
constexpr int kFlagSubFirst = 4;  // first member of its cascade subgroup

struct PlanSmem {
  int S[kMaxSeqs];          // seq_len, -1 if the row is invalid
  int L[kMaxSeqs];
  int Q0[kMaxSeqs];         // first query token
  int lcp[kMaxSeqs];        // leading pages equal to the previous row's
  int gid[kMaxSeqs];        // run (group) id
  int grp_pages[kMaxSeqs];  // per group: shared full pages
  int grp_ndec[kMaxSeqs];   // per group: decode rows
  int grp_base[kMaxSeqs];   // per group: smallest member rank
  int mrank[kMaxSeqs];      // member rank (cascade member array index)
  int own_pb[kMaxSeqs];     // first page of the row's own decode range
  int n_cs[kMaxSeqs];       // cascade splits covering the row
  int part_off[kMaxSeqs];
  int item_off[kMaxSeqs];   // decode records
  int sg_off[kMaxSeqs];     // cascade records (subgroup-first rows only)
  int tile_off[kMaxSeqs];   // append records
  int sub_first_idx[kMaxSeqs];  // first member index of the row's subgroup
  int sub_n[kMaxSeqs];          // members in the row's subgroup
  int app_row[kMaxSeqs];        // append rows, longest first (row of rank k)
  int app_off[kMaxSeqs];        // first append record of the rank-k row
  unsigned char kind[kMaxSeqs];   // 0 none / invalid, 1 decode, 2 append
  unsigned char flags[kMaxSeqs];
  ScanBuf sb;
  int bad_global;
  int split_pages;
};

template <int NT>
__global__ void __launch_bounds__(NT, 1) plan_kernel(AttnParams p) {
  constexpr int kWarps = NT / 32;
  extern __shared__ __align__(16) uint8_t plan_smem_raw[];
  PlanSmem& sm = *reinterpret_cast<PlanSmem*>(plan_smem_raw);
  PlanHeader* hdr = header(p);
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int B = p.num_seqs;
  const int tile_tok = p.append_tile_tok;
  const int sub_cap = 32 / p.group;  // rows per cascade item (32 query vectors)

  if (tid == 0) {
    const int bad = (p.qsl[0] != 0 || p.qsl[B] != p.total_q) ? 1 : 0;
    sm.bad_global = bad;
    if (bad) atomicOr(&hdr->status, kStatusBadLengths);
  }
  __syncthreads();
  if (sm.bad_global) {
    grid_dep_wait();  // nothing of this call ends before the prefix scan
    if (tid == 0) {
      hdr->n_decode = hdr->n_cascade = hdr->n_append = hdr->n_merge = 0;
      hdr->n_parts = 0;
      hdr->append_ticket = hdr->decode_ticket = hdr->cascade_ticket = 0;
    }
    return;
  }

  // ---- phase 1: per-row kind and lengths
  for (int r = tid; r < B; r += NT) {
    const int q0 = p.qsl[r], q1 = p.qsl[r + 1];
    const int len = q1 - q0, s = p.seq_lens[r];
    const bool bad = len < 0 || s < len || s > p.max_pages * kPage;
    if (bad) atomicOr(&hdr->status, kStatusBadLengths);
    // decode-only calls (fp8 pools) report and skip append rows
    const bool skip = !bad && p.decode_only && len > 1;
    if (skip) atomicOr(&hdr->status, kStatusUnsupportedRow);
    sm.S[r] = (bad || skip) ? -1 : s;
    sm.L[r] = (bad || skip) ? 0 : len;
    sm.Q0[r] = q0;
    sm.kind[r] = (bad || skip) ? 0 : (len == 0 ? 0 : (len == 1 ? 1 : 2));
    sm.lcp[r] = 0;
    sm.grp_pages[r] = 0x7fffffff;
    sm.grp_ndec[r] = 0;
    sm.grp_base[r] = 0x7fffffff;
    sm.flags[r] = 0;
  }
  __syncthreads();

  // ---- phase 2: shared-prefix groups (full-context calls only)
  // lcp[r] = leading physical pages row r shares with row r - 1 (full pages
  // of both), scanned beforehand by lcp_kernel across the whole GPU. The
  // planner may have been launched while that scan ran (phase 1 reads only
  // the caller's arrays): wait for it here.
  grid_dep_wait();
  const bool cascade = p.cascade_enabled && p.window <= 0;
  if (cascade) {
    const int* lcp_ws = reinterpret_cast<const int*>(p.ws + p.lay.lcp);
    for (int r = tid; r < B; r += NT) {
      const int sa = r > 0 ? sm.S[r - 1] : -1, sb = sm.S[r];
      sm.lcp[r] = (sa < 0 || sb < 0) ? 0 : min(lcp_ws[r], min(sa, sb) / kPage);
    }
  }
  __syncthreads();
  // group id = (number of run starts up to and including r) - 1
  for (int r = tid; r < B; r += NT)
    sm.gid[r] = (r == 0 || !cascade || sm.lcp[r] < kMinSharedPages) ? 1 : 0;
  __syncthreads();
  {
    int st[R];
#pragma unroll
    for (int i = 0; i < R; ++i) {
      const int r = tid * R + i;
      st[i] = r < B ? sm.gid[r] : 0;
    }
    __syncthreads();
    int total, sum = 0;
#pragma unroll
    for (int i = 0; i < R; ++i) sum += st[i];
    int base = cta_scan<NT>(sum, &total, sm.sb);
#pragma unroll
    for (int i = 0; i < R; ++i) {
      const int r = tid * R + i;
      base += st[i];
      if (r < B) sm.gid[r] = base - 1;
    }
  }
  __syncthreads();
  if (cascade) {
    for (int r = tid; r < B; r += NT) {
      const int g = sm.gid[r];
      if (r > 0 && sm.gid[r - 1] == g) atomicMin(&sm.grp_pages[g], sm.lcp[r]);
      if (sm.kind[r] == 1) {
        atomicMin(&sm.grp_pages[g], sm.S[r] / kPage);
        atomicAdd(&sm.grp_ndec[g], 1);
      }
    }
  }
  __syncthreads();
  // members: decode rows of a group with >= 2 decode rows and a long enough prefix
  for (int r = tid; r < B; r += NT) {
    int m = 0;
    if (cascade && sm.kind[r] == 1) {
      const int g = sm.gid[r];
      m = (sm.grp_ndec[g] >= 2 && sm.grp_pages[g] >= kMinSharedPages) ? 1 : 0;
    }
    sm.mrank[r] = m;
    if (m) sm.flags[r] |= kFlagMember;
  }
  __syncthreads();
  scan_rows<NT>(sm.mrank, B, sm.sb);
  for (int r = tid; r < B; r += NT)
    if (sm.flags[r] & kFlagMember) atomicMin(&sm.grp_base[sm.gid[r]], sm.mrank[r]);
  __syncthreads();

  // ---- phase 3: split length
  int w_m = 0, w_lb = 0;
  for (int r = tid; r < B; r += NT) {
    sm.own_pb[r] = 0;
    sm.n_cs[r] = 0;
    sm.sub_first_idx[r] = 0;
    sm.sub_n[r] = 0;
    if (sm.kind[r] != 1) continue;
    const int S = sm.S[r];
    const int first_key = p.window > 0 ? max(0, S - p.window) : 0;
    const int pe = cdiv(S, kPage);
    int pb = first_key / kPage;
    int gp = 0;
    if (sm.flags[r] & kFlagMember) {
      const int g = sm.gid[r];
      const int nd = sm.grp_ndec[g];
      gp = sm.grp_pages[g];
      pb = gp;
      const int nsub = cdiv(nd, sub_cap);
      const int idx = sm.mrank[r] - sm.grp_base[g];
      const int sub = idx * nsub / nd;
      const int first = cdiv(sub * nd, nsub), next = cdiv((sub + 1) * nd, nsub);
      sm.sub_first_idx[r] = sm.grp_base[g] + first;
      sm.sub_n[r] = next - first;
      if (idx == first) sm.flags[r] |= kFlagSubFirst;
    }
    sm.own_pb[r] = pb;
    sm.n_cs[r] = gp;  // shared pages for now; split count after C is known
    const int own = pe - pb;
    w_m += own + gp;
    w_lb += own + ((sm.flags[r] & kFlagSubFirst) ? gp : 0);
  }
  int tot_wm, tot_wlb;
  cta_scan<NT>(w_m, &tot_wm, sm.sb);
  cta_scan<NT>(w_lb, &tot_wlb, sm.sb);
  const int c_bound = max(1, cdiv(tot_wm, kSplitBudget));
  int C;
  if (p.forced_split_pages > 0) {
    C = max(p.forced_split_pages, c_bound);
  } else {
    // W = (page, kv head) blocks per decode warp. A split of C pages costs a
    // fixed overhead of about 12 pages' time (query setup, ring ramp, the
    // partial's write and merge) and leaves a tail of about C / 2 pages at the
    // end, so the time per warp ~ W + 12 W / C + C / 2 is least at
    // C = sqrt(24 W) (measured optimum 64 pages at W = 162 and 384-512 at
    // W = 4441 for bf16 pages, 48 at W = 121 and 256 at W = 3330 for fp8).
    const float w = (float)tot_wlb * (float)p.num_kv_heads / (float)max(p.total_warps_hint, 1);
    const int c_opt = (int)(sqrtf(24.f * w) + 0.5f);
    C = max(kMinSplitPages, max(c_opt, c_bound));
  }

  // ---- phase 4: per-row counts -> offsets
  for (int r = tid; r < B; r += NT) {
    int n_own = 0, n_cs = 0, parts = 0, tiles = 0, sg = 0, direct = 0;
    if (sm.kind[r] == 1) {
      const int pe = cdiv(sm.S[r], kPage);
      n_own = cdiv(pe - sm.own_pb[r], C);
      const bool member = sm.flags[r] & kFlagMember;
      n_cs = member ? cdiv(sm.n_cs[r], C) : 0;
      parts = n_own + n_cs;
      direct = (!member && parts == 1) ? 1 : 0;
      if (direct) sm.flags[r] |= kFlagDirect;
      if (sm.flags[r] & kFlagSubFirst) sg = n_cs;
    } else if (sm.kind[r] == 2) {
      tiles = cdiv(sm.L[r], tile_tok);
    }
    sm.n_cs[r] = n_cs;
    sm.part_off[r] = direct ? 0 : parts;
    sm.item_off[r] = n_own;
    sm.sg_off[r] = sg;
    sm.tile_off[r] = tiles;
  }
  __syncthreads();
  const int tot_parts = scan_rows<NT>(sm.part_off, B, sm.sb);
  const int tot_items = scan_rows<NT>(sm.item_off, B, sm.sb);
  const int tot_cascade = scan_rows<NT>(sm.sg_off, B, sm.sb);
  const int tot_tiles = scan_rows<NT>(sm.tile_off, B, sm.sb);

  // ---- append rows, longest first: the persistent append kernel takes its
  // items in record order, so it starts with the rows that have the most
  // keys (the longest items) and ends on short ones, which shortens its tail
  // (a list-scheduling model of the 256-row mixed batch: 2.0 % -> 0.6 % idle
  // at the end). Ties keep row order; above kMaxRanked rows the ranking's
  // n^2 comparisons are skipped and row order stays.
  constexpr int kMaxRanked = 512;
  for (int r = tid; r < B; r += NT) sm.app_off[r] = sm.kind[r] == 2 ? 1 : 0;
  __syncthreads();
  const int n_app = scan_rows<NT>(sm.app_off, B, sm.sb);
  for (int r = tid; r < B; r += NT)
    if (sm.kind[r] == 2) sm.app_row[sm.app_off[r]] = r;  // compact, row order
  __syncthreads();
  if (n_app <= kMaxRanked) {
    for (int i = tid; i < n_app; i += NT) {
      const int r = sm.app_row[i], Sr = sm.S[r];
      int rank = 0;
      for (int j = 0; j < n_app; ++j) {
        const int q = sm.app_row[j], Sq = sm.S[q];
        rank += (Sq > Sr || (Sq == Sr && q < r)) ? 1 : 0;
      }
      sm.app_off[rank] = r;  // app_off as scratch: row of each rank
    }
    __syncthreads();
    for (int i = tid; i < n_app; i += NT) sm.app_row[i] = sm.app_off[i];
    __syncthreads();
  }
  for (int i = tid; i < n_app; i += NT) sm.app_off[i] = cdiv(sm.L[sm.app_row[i]], tile_tok);
  __syncthreads();
  scan_rows<NT>(sm.app_off, n_app, sm.sb);

  const bool overflow = tot_items > p.lay.max_decode || tot_cascade > p.lay.max_cascade ||
                        tot_tiles > p.lay.max_append || tot_parts > p.lay.max_parts;
  if (overflow) {
    if (tid == 0) {
      atomicOr(&hdr->status, kStatusPlanOverflow);
      hdr->n_decode = hdr->n_cascade = hdr->n_append = hdr->n_merge = 0;
      hdr->n_parts = 0;
      hdr->append_ticket = hdr->decode_ticket = hdr->cascade_ticket = 0;
    }
    return;
  }

  DecodeItem* ditems = reinterpret_cast<DecodeItem*>(p.ws + p.lay.decode_items);
  CascadeItem* citems = reinterpret_cast<CascadeItem*>(p.ws + p.lay.cascade_items);
  CascadeMember* members = reinterpret_cast<CascadeMember*>(p.ws + p.lay.members);
  AppendItem* aitems = reinterpret_cast<AppendItem*>(p.ws + p.lay.append_items);
  MergeRow* mrows = reinterpret_cast<MergeRow*>(p.ws + p.lay.merge_rows);

  // ---- phase 5: per-row records (merge rows, cascade members)
  int is_merge_cnt = 0;
  {
    // merge rows get consecutive indices: reuse lcp[] as the scan buffer
    for (int r = tid; r < B; r += NT)
      sm.lcp[r] = (sm.kind[r] == 1 && !(sm.flags[r] & kFlagDirect)) ? 1 : 0;
    __syncthreads();
    is_merge_cnt = scan_rows<NT>(sm.lcp, B, sm.sb);
  }
  for (int r = tid; r < B; r += NT) {
    if (sm.kind[r] != 1) continue;
    const int parts = (r + 1 < B ? sm.part_off[r + 1] : tot_parts) - sm.part_off[r];
    if (!(sm.flags[r] & kFlagDirect)) {
      MergeRow m;
      m.token = sm.Q0[r];
      m.n_parts = parts;
      m.part_off = sm.part_off[r];
      m.pad = 0;
      mrows[sm.lcp[r]] = m;
    }
    if (sm.flags[r] & kFlagMember) {
      CascadeMember cm;
      cm.row = r;
      cm.token = sm.Q0[r];
      cm.part_off = sm.part_off[r];
      cm.pad = 0;
      members[sm.mrank[r]] = cm;
    }
  }

  // ---- phase 6: split records, all threads in parallel
  for (int e = tid; e < tot_items; e += NT) {
    const int r = owner_row(sm.item_off, B, e);
    const int k = e - sm.item_off[r];
    const int S = sm.S[r];
    const int pe = cdiv(S, kPage);
    DecodeItem it;
    it.row = r;
    it.token = sm.Q0[r];
    it.seq_len = S;
    it.first_key = p.window > 0 ? max(0, S - p.window) : 0;
    it.page_begin = sm.own_pb[r] + k * C;
    it.page_end = min(pe, sm.own_pb[r] + (k + 1) * C);
    it.slot = (sm.flags[r] & kFlagDirect) ? -1 : sm.part_off[r] + sm.n_cs[r] + k;
    it.pad = 0;
    ditems[e] = it;
  }
  // Cascade records of one group go split-major: (split k, subgroup s) at
  // the group's base + k * nsub + s, so the subgroups of a group (g = 8:
  // two of 4 rows) read the same pages within a few tickets of each other
  // and the second read of each page is an L2 hit, not a second HBM read.
  for (int e = tid; e < tot_cascade; e += NT) {
    const int r = owner_row(sm.sg_off, B, e);
    const int k = e - sm.sg_off[r];
    const int g = sm.gid[r];
    const int gp = sm.grp_pages[g];
    const int nd = sm.grp_ndec[g], nsub = cdiv(nd, sub_cap);
    const int s = (sm.mrank[r] - sm.grp_base[g]) * nsub / nd;
    const int dst = sm.sg_off[r] - s * sm.n_cs[r] + k * nsub + s;
    CascadeItem c;
    c.member_off = sm.sub_first_idx[r];
    c.n_members = sm.sub_n[r];
    c.page_begin = k * C;
    c.page_end = min(gp, (k + 1) * C);
    c.split = k;
    c.first_row = r;
    c.pad0 = c.pad1 = 0;
    citems[dst] = c;
  }
  for (int e = tid; e < tot_tiles; e += NT) {
    const int i = owner_row(sm.app_off, n_app, e);
    const int r = sm.app_row[i];
    const int S = sm.S[r], L = sm.L[r];
    const int k = cdiv(L, tile_tok) - 1 - (e - sm.app_off[i]);  // a row's last (longest) tile first
    AppendItem a;
    a.row = r;
    a.token_begin = sm.Q0[r] + k * tile_tok;
    a.n_tok = min(tile_tok, L - k * tile_tok);
    a.seq_len = S;
    a.pos_begin = S - L + k * tile_tok;
    a.key_begin = p.window > 0 ? max(0, a.pos_begin - p.window + 1) : 0;
    a.key_end = a.pos_begin + a.n_tok;
    a.pad = 0;
    aitems[e] = a;
  }
  if (tid == 0) {
    hdr->n_decode = tot_items;
    hdr->n_cascade = tot_cascade;
    hdr->n_append = tot_tiles;
    hdr->n_merge = is_merge_cnt;
    hdr->split_pages = C;
    hdr->n_parts = tot_parts;
    hdr->append_ticket = hdr->decode_ticket = hdr->cascade_ticket = 0;
  }
}

// One warp per adjacent row pair (r - 1, r): the number of leading block-table
// entries the two rows share, over the pages full in both (lengths outside
// the table count as none). 512 entries per step: 16 loads of each row per
// lane in flight, one ballot per 32. Writes lcp[r] (lcp[0] = 0).
constexpr int kLcpWarps = 8;
constexpr int kLcpPerLane = 16;

__global__ void __launch_bounds__(kLcpWarps * 32) lcp_kernel(const AttnParams p) {
  grid_dep_launch();  // the planner may start its first phase meanwhile
  const int lane = threadIdx.x & 31;
  const int r = blockIdx.x * kLcpWarps + (threadIdx.x >> 5);
  int* lcp = reinterpret_cast<int*>(p.ws + p.lay.lcp);
  if (r >= p.num_seqs) return;
  if (r == 0) {
    if (lane == 0) lcp[0] = 0;
    return;
  }
  const int cap = p.max_pages * kPage;
  const int sa = __ldg(p.seq_lens + r - 1), sb = __ldg(p.seq_lens + r);
  const int lim = (sa < 0 || sb < 0 || sa > cap || sb > cap) ? 0 : min(sa, sb) / kPage;
  const int* ba = p.block_table + (size_t)(r - 1) * p.max_pages;
  const int* bb = p.block_table + (size_t)r * p.max_pages;
  int n = 0;
  for (int base = 0; base < lim; base += 32 * kLcpPerLane) {
    int va[kLcpPerLane], vb[kLcpPerLane];
#pragma unroll
    for (int j = 0; j < kLcpPerLane; ++j) {
      const int i = base + 32 * j + lane;
      va[j] = i < lim ? __ldg(ba + i) : 0;
      vb[j] = i < lim ? __ldg(bb + i) : 1;
    }
    bool stop = false;
#pragma unroll
    for (int j = 0; j < kLcpPerLane; ++j) {
      const unsigned m = __ballot_sync(0xffffffffu, va[j] == vb[j]);
      if (!stop) {
        if (m == 0xffffffffu) {
          n += 32;
        } else {
          n += __ffs(~m) - 1;
          stop = true;
        }
      }
    }
    if (stop) break;
  }
  if (lane == 0) lcp[r] = min(n, lim);
}

cudaError_t launch_plan(const AttnParams& p, cudaStream_t stream, bool programmatic) {
  static_assert(sizeof(PlanSmem) < 200 * 1024, "planner shared memory");
  const bool scan = p.cascade_enabled && p.window <= 0 && p.num_seqs > 0;
  if (scan) {
    lcp_kernel<<<(p.num_seqs + kLcpWarps - 1) / kLcpWarps, kLcpWarps * 32, 0, stream>>>(p);
    const cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
  }
  // After the prefix scan (and only then: an earlier grid of the caller's
  // may write what phase 1 reads) the planner may be launched
  // programmatically, so that its launch and first phase overlap the scan.
  // Fewer threads for small batches: every phase ends in a CTA barrier, and
  // barriers over 8 warps are cheaper than over 32.
  const bool small = p.num_seqs <= R * 256;
  LaunchCfg lc(dim3(1), dim3(small ? 256 : kPlanThreads), sizeof(PlanSmem), stream, programmatic && scan);
  return small ? cudaLaunchKernelEx(&lc.cfg, plan_kernel<256>, p) : cudaLaunchKernelEx(&lc.cfg, plan_kernel<kPlanThreads>, p);
}

cudaError_t prepare_plan_kernel() {
  // every kernel of the library asks for the largest shared-memory carveout,
  // so an SM never has to be reconfigured between them and a decode CTA can
  // share an SM with an append CTA
  cudaError_t e = cudaFuncSetAttribute(plan_kernel<256>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)sizeof(PlanSmem));
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(plan_kernel<256>, cudaFuncAttributePreferredSharedMemoryCarveout,
                             cudaSharedmemCarveoutMaxShared);
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(plan_kernel<kPlanThreads>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)sizeof(PlanSmem));
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(plan_kernel<kPlanThreads>, cudaFuncAttributePreferredSharedMemoryCarveout,
                             cudaSharedmemCarveoutMaxShared);
  return e;
}

}  // namespace mcpu
