// One tournament round and the shared-prefix segment rebuild in a single launch.
//
// The Tournament of Algorithm 1 (Eq. 2, Case 1 under capacity; Eq. 3, Case 2 at
// capacity) ranks the active traces by running mean, prunes the bottom K and branches the
// top eligible traces; a branched child inherits its parent's KV by taking the parent's
// block table (Section 3.1, after Eq. 3), and a pruned trace frees only the pages nobody
// else holds.  After the round the grouped attention path needs the new shared-prefix
// segments.  All of it runs here as one persistent grid (one CTA of 1024 threads per SM
// at most, so every CTA is resident at once) in four phases separated by bounded grid
// barriers:
//
//   1. tournament: every CTA ranks the active slots redundantly (bitonic sort of 64-bit
//      keys, shuffles for the strides inside a warp) and derives the same routing; the
//      parents are spread over the CTAs, and each forks its children's block tables:
//      a page that c of the parent's children newly hold gets one +c, each child drops
//      the references of its old table, and the children's per-slot state is written.
//      Why no page is freed too early: a page held by a surviving beam keeps that
//      reference for the whole round (survivors are never pruned), so only pages held by
//      pruned beams alone can reach zero, and no child takes such a page.
//   2. segments: a group of threads per beam walks its table.  A segment is a maximal run
//      of full pages with one sharer set of at least group_min beams; along one table the
//      sharer count (the refcount) never increases and changes exactly where the sharer
//      set changes, so segment starts are refcount change points.  The first member of a
//      segment to reach its first page claims it (an atomic maximum on a per-page word
//      stamped with the rebuild generation, a counter the kernel itself advances, so a
//      replayed CUDA graph gets a fresh one) and publishes its id; the other members wait
//      for the id (bounded) and append themselves to the member list.
//   3. work list, part 1: the token split of the grouped work units (from the segments'
//      totals) and a histogram of unit lengths.
//   4. work list, part 2: units laid out longest first, and every beam's record offsets.
//
// Segment ids and member order follow atomics, but every output row of the grouped
// kernel is computed independently of its position, so results do not depend on them.
// Without a tournament (after seeding, a release or gb_fork_slots) the kernel runs phases
// 2-4 only.  A barrier that waits too long records GB_ERR_TIMEOUT and the CTA returns.
#include "internal.cuh"
#include "ptx.cuh"

namespace gb {

constexpr int kTourThreads = 1024;
constexpr int kSegLenBuckets = 256;  // work units sorted by length in 128-token tiles (longer ones share the last bucket)

#ifndef GB_SEG_UNITS_PCT
#define GB_SEG_UNITS_PCT 200  // grouped work units aimed at per multiprocessor, in percent
#endif

struct TourArgs {
  int prune;               // 1: run the tournament first
  int C, K, fanout, warmup;
  const uint8_t* elig;     // caller's eligibility mask or nullptr
  int* parent_out;
  uint8_t* pruned_out;
  unsigned* lineage_out;
};

// Unsigned key whose ascending order is: larger mean first, +0 == -0, NaN last.
__device__ __forceinline__ unsigned rank_key(float m) {
  if (isnan(m)) return 0xffffffffu;
  if (m == 0.f) m = 0.f;
  const unsigned u = __float_as_uint(m);
  const unsigned asc = (u & 0x80000000u) ? ~u : (u | 0x80000000u);
  return ~asc;
}

// Grid-wide barrier over a grid whose CTAs are all resident.  The arrival counter only ever
// grows: barrier n of a grid of G CTAs is passed once it reaches the next multiple of G above
// a CTA's own arrival, so the last arrival releases everyone with no reset (the count is a
// multiple of G between launches, which every launch of this kernel on the pool keeps).
__device__ bool grid_sync(const PoolView& v, int* s_fail) {
  __syncthreads();
  if (threadIdx.x == 0 && *s_fail == 0) {
    fence_acq_rel_gpu();  // this CTA's writes before its arrival
    const unsigned G = gridDim.x;
    const unsigned old = atomicAdd(reinterpret_cast<unsigned*>(v.ctl + kCtlBarCount), 1u);
    const unsigned target = (old / G + 1) * G;
    volatile unsigned* cnt = reinterpret_cast<volatile unsigned*>(v.ctl + kCtlBarCount);
    if (old + 1 != target) {
      const uint64_t t0 = globaltimer_ns();
      for (unsigned it = 1; (int)(*cnt - target) < 0; ++it) {
        if ((it & 63) == 0 && globaltimer_ns() - t0 > kWaitLimitNs) {
          set_status(v.ctl, GB_ERR_TIMEOUT);
          *s_fail = 1;
          break;
        }
      }
    }
    fence_acq_rel_gpu();  // the other CTAs' writes after the barrier
  }
  __syncthreads();
  return *s_fail == 0;
}

// Group-wide exclusive scan (groups of `tpb` consecutive threads, tpb a power of two >= 32)
// through a block-wide scan: the group's prefix is the block prefix minus that of its first
// thread.  Called by every thread of the block; *group_total gets the group's sum.
__device__ __forceinline__ int group_exclusive_scan(int x, int tpb, int* tmp, int* s_pref, int* group_total) {
  int total;
  const int pre = block_exclusive_scan(x, tmp, &total);
  s_pref[threadIdx.x] = pre;
  __syncthreads();
  const int first = threadIdx.x & ~(tpb - 1);
  const int next = first + tpb;
  const int base = s_pref[first];
  *group_total = (next < (int)blockDim.x ? s_pref[next] : total) - base;
  __syncthreads();
  return pre - base;
}

__global__ void __launch_bounds__(kTourThreads, 1) k_tournament(PoolView v, TourArgs a) {
  pdl_wait();
  __shared__ unsigned long long s_keys[kMaxBeams];
  __shared__ int ord[kMaxBeams];      // rank -> slot
  __shared__ int blist[kMaxBeams];    // eligible parents in rank order
  __shared__ int cslot[kMaxBeams];    // child k -> slot
  __shared__ int childof[kMaxBeams];  // slot -> child index or -1
  __shared__ int s_oldn[kMaxBeams];   // child k -> table entries its slot held before the fork
  __shared__ unsigned char s_act[kMaxBeams], s_elig[kMaxBeams], s_pruned[kMaxBeams];
  __shared__ int s_pref[kTourThreads];
  __shared__ int tmp[33];
  __shared__ int s_fail, s_nchild;
  __shared__ unsigned s_lin0;
  __shared__ unsigned long long s_gen;
  // phase 2 (per group of threads: up to 32 groups)
  __shared__ int s_low[32], s_cap[32], s_nst[32], s_carry_g[32];
  __shared__ int s_start[32][kMaxSegDepth], s_spage[32][kMaxSegDepth];
  // phases 3-4
  __shared__ int s_hist[kSegLenBuckets];
  __shared__ int s_split, s_total;
  __shared__ int s_rowtok, s_tiletok, s_segtok;  // this CTA's share of the segment totals
  __shared__ int s_freed, s_minword;              // pages this CTA freed, lowest freed bitmap word

  const int tid = threadIdx.x;
  const int cap = v.max_beams;
  // The slot's state for the ranking, loaded first and together.
  const bool in = a.prune && tid < cap;
  const int act_w = in ? v.active[tid] : 0;
  const int gen_w = in ? v.gen[tid] : 0;
  const float mean_w = in ? v.mean[tid] : 0.f;
  const int elig_w = (in && a.elig != nullptr) ? a.elig[tid] : 1;
  if (tid == 0) {
    s_fail = 0;
    s_nchild = 0;
    s_rowtok = s_tiletok = s_segtok = 0;
    s_freed = 0;
    s_minword = 0x7fffffff;
    s_lin0 = (unsigned)v.ctl[kCtlNextLineage];
  }
  if (blockIdx.x == 0 && tid < 2 * kSegLenBuckets) v.seg_hist[tid] = 0;
  if (blockIdx.x == 0 && tid == 0) {
    v.ctl[kCtlSegGen] += 1;  // this rebuild's generation, read by every CTA after the first barrier
    v.ctl[kCtlSegAlloc] = 0;  // segments (high word of the pair) and member slots (low word)
    v.ctl[kCtlSegAlloc + 1] = 0;
    v.ctl[kCtlSegRowTok] = 0;
    v.ctl[kCtlSegTileTok] = 0;
    v.ctl[kCtlSegTok] = 0;
  }
  __syncthreads();

  // ---- 1. tournament ---------------------------------------------------------------------
  if (a.prune) {
    const bool act = act_w != 0;
    const bool elig = act && gen_w >= a.warmup && elig_w != 0;
    s_act[tid] = act;
    s_elig[tid] = elig;
    s_pruned[tid] = 0;
    childof[tid] = -1;
    int N;
    const int pos = block_exclusive_scan(act ? 1 : 0, tmp, &N);
    s_keys[tid] = ~0ull;
    __syncthreads();
    if (act) s_keys[pos] = ((unsigned long long)rank_key(mean_w) << 32) | (unsigned)tid;
    __syncthreads();
    // Rank (ascending keys; the slot in the low word makes them distinct): each warp sorts its
    // 32 keys in registers (bitonic, by shuffles), then a key's rank is its position in its
    // warp's list plus, for every other list, the number of keys there below it (a binary
    // search over 32 sorted keys; four lists at a time).
    const int nl = (N + 31) >> 5, lane = tid & 31, wl = tid >> 5;
    if (wl < nl) {
      unsigned long long my = s_keys[tid];  // ~0 past the N keys
      for (int k = 2; k <= 32; k <<= 1)
        for (int j = k >> 1; j > 0; j >>= 1) {
          const unsigned long long other = __shfl_xor_sync(0xffffffffu, my, j);
          const bool asc = (lane & k) == 0, lower = (lane & j) == 0;
          my = (asc == lower) ? (my < other ? my : other) : (my > other ? my : other);
        }
      s_keys[tid] = my;
      asm volatile("bar.sync 1, %0;" ::"r"(nl * 32) : "memory");
      if (my != ~0ull) {
        int rank = lane;
        for (int l0 = 0; l0 < nl; l0 += 4) {
          int pos[4] = {0, 0, 0, 0};
#pragma unroll
          for (int st = 16; st > 0; st >>= 1)
#pragma unroll
            for (int u = 0; u < 4; ++u)
              if (l0 + u < nl && s_keys[32 * (l0 + u) + pos[u] + st - 1] < my) pos[u] += st;
#pragma unroll
          for (int u = 0; u < 4; ++u)
            if (l0 + u < nl && l0 + u != wl) rank += pos[u] + (s_keys[32 * (l0 + u) + pos[u]] < my ? 1 : 0);
        }
        ord[rank] = (int)(my & 0xffffffffu);
      }
    }
    __syncthreads();
    // Routing (identical in every CTA).
    const int f1 = a.fanout - 1;
    int nchild = 0, kase = 0;
    if (N > 0 && N < a.C) {
      // Case 1 (Eq. 2): the top min(C - N, |B|) eligible traces, one child each, into vacant slots.
      kase = 1;
      const bool f = tid < N && s_elig[ord[tid]];
      int nb;
      const int pb = block_exclusive_scan(f ? 1 : 0, tmp, &nb);
      if (f) blist[pb] = ord[tid];
      nchild = min(a.C - N, nb);
      const bool vac = tid < cap && !act;
      int nv;
      const int pv = block_exclusive_scan(vac ? 1 : 0, tmp, &nv);
      if (vac && pv < nchild) cslot[pv] = tid;
    } else if (N > 0) {
      // Case 2 (Eq. 3, fan-out f; N = C): prune the bottom K_eff, branch the top eligible survivors.
      kase = 2;
      const int Kc = a.K < 0 ? 0 : (a.K > N ? N : a.K);
      const int nsurv = N - Kc;
      const bool f = tid < nsurv && s_elig[ord[tid]];
      int nb;
      const int pb = block_exclusive_scan(f ? 1 : 0, tmp, &nb);
      if (f) blist[pb] = ord[tid];
      const long long cap_children = (long long)f1 * nb;
      nchild = (int)(Kc < cap_children ? Kc : cap_children);
      if (tid >= N - nchild && tid < N) s_pruned[ord[tid]] = 1;
      __syncthreads();
      const bool pr = tid < cap && s_pruned[tid];
      int np;
      const int pp = block_exclusive_scan(pr ? 1 : 0, tmp, &np);
      if (pr) cslot[pp] = tid;
    }
    __syncthreads();
    if (tid < nchild) childof[cslot[tid]] = tid;
    if (tid == 0) s_nchild = nchild;
    __syncthreads();
    // Parent j has children [j * per, min((j + 1) * per, nchild)): per = 1 in Case 1, f - 1 in Case 2.
    const int per = kase == 2 ? f1 : 1;
    const int npar = (nchild + per - 1) / per;
    const unsigned lin0 = s_lin0;

    // Children share their parents' partial tail pages until the next step's planner copies them.
    if (blockIdx.x == 0 && tid == 0 && nchild > 0) v.ctl[kCtlTailShared] = 1;
    // Outputs (CTA 0): parent_of, pruned flags, lineage ids after the round.
    if (blockIdx.x == 0 && tid < cap) {
      const int k = childof[tid];
      if (a.parent_out) a.parent_out[tid] = k >= 0 ? blist[k / per] : (s_act[tid] ? tid : -1);
      if (a.pruned_out) a.pruned_out[tid] = s_pruned[tid];
      if (a.lineage_out) a.lineage_out[tid] = k >= 0 ? lin0 + k : v.lineage[tid];
    }
    // Fork: this CTA's parents, each by its own group of threads (ppc parents at a time).  For
    // table index i of parent p, each child c either already holds page tp[i] (nothing
    // changes) or drops its old page and takes tp[i]; the new references of one parent's page
    // are added at once.  A page whose last reference drops is marked free in the bitmap; the
    // CTA's count of freed pages and lowest freed bitmap word are kept in shared memory and
    // added to the pool's counters once per CTA.
    // The children's table lengths before the fork, one load per child for all its entries.
    for (int c = tid; c < nchild; c += blockDim.x) {
      const int sl = cslot[c];
      s_oldn[c] = s_act[sl] ? (v.seq_len[sl] + v.P - 1) / v.P : 0;
    }
    __syncthreads();
    const int mine = npar > (int)blockIdx.x ? (npar - 1 - (int)blockIdx.x) / (int)gridDim.x + 1 : 0;
    int ppc = 1;
    while (ppc < 32 && ppc < mine) ppc <<= 1;
    const int tpp = kTourThreads / ppc, fg = tid / tpp, ft = tid % tpp;
    for (int j = blockIdx.x + fg * gridDim.x; j < npar; j += ppc * gridDim.x) {
      const int p = blist[j];
      const int k0 = j * per, k1 = min(k0 + per, nchild);
      const int new_n = (v.seq_len[p] + v.P - 1) / v.P;
      int m = new_n;
      for (int c = k0; c < k1; ++c) m = max(m, s_oldn[c]);
      const int* tp = v.tables + (size_t)p * v.max_pages;
      for (int i = ft; i < m; i += tpp) {
        const int nw = i < new_n ? tp[i] : -1;
        int add = 0;
        // Four children at a time: their old entries, then their reference drops, are
        // issued together rather than one child after another.
        for (int c0 = k0; c0 < k1; c0 += 4) {
          int old[4], dec[4];
#pragma unroll
          for (int u = 0; u < 4; ++u) {
            const int c = c0 + u;
            old[u] = nw;  // no child: nothing changes
            if (c < k1) old[u] = i < s_oldn[c] ? v.tables[(size_t)cslot[c] * v.max_pages + i] : -1;
          }
#pragma unroll
          for (int u = 0; u < 4; ++u) dec[u] = (old[u] != nw && old[u] >= 0) ? atomicSub(&v.refcnt[old[u]], 1) : 0;
#pragma unroll
          for (int u = 0; u < 4; ++u) {
            if (old[u] == nw) continue;
            if (nw >= 0) ++add;
            if (dec[u] == 1) {  // the page's last reference: it is free
              atomicOr(&v.free_bits[old[u] >> 5], 1u << (old[u] & 31));
              atomicMin(&s_minword, old[u] >> 5);
              atomicAdd(&s_freed, 1);
            }
            if (i < new_n) v.tables[(size_t)cslot[c0 + u] * v.max_pages + i] = nw;
          }
        }
        if (add > 0) atomicAdd(&v.refcnt[nw], add);
      }
    }
    __syncthreads();  // every thread has read the children's old lengths
    // The children's per-slot state, for the parents this CTA forked.
    for (int c = tid; c < nchild; c += blockDim.x) {
      const int j = c / per;
      if (j % (int)gridDim.x != (int)blockIdx.x) continue;
      const int sl = cslot[c], p = blist[j];
      v.seq_len[sl] = v.seq_len[p];
      v.mean[sl] = v.mean[p];
      v.nsteps[sl] = v.nsteps[p];
      v.gen[sl] = 0;
      v.active[sl] = 1;
      v.lineage[sl] = lin0 + c;
    }
    __syncthreads();
    if (tid == 0 && s_freed > 0) {
      atomicAdd(&v.ctl[kCtlFree], s_freed);
      atomicMin(&v.ctl[kCtlCursor], s_minword);
    }
  }
  if (!v.grouped) {
    // No grouped path: no segments to rebuild.  The lineage counter moves on once every CTA
    // has read it, which without a barrier the last CTA to finish guarantees.
    __shared__ int s_last;
    __threadfence();
    __syncthreads();
    if (tid == 0) s_last = atomicAdd(&v.ctl[kCtlDone], 1) == (int)gridDim.x - 1;
    __syncthreads();
    if (s_last && tid == 0) {
      v.ctl[kCtlNextLineage] = (int)(s_lin0 + s_nchild);
      v.ctl[kCtlDone] = 0;
    }
    pdl_launch_dependents();
    return;
  }
  if (!grid_sync(v, &s_fail)) return;
  if (blockIdx.x == 0 && tid == 0 && a.prune) v.ctl[kCtlNextLineage] = (int)(s_lin0 + s_nchild);
  if (tid == 0) s_gen = (unsigned long long)(unsigned)v.ctl[kCtlSegGen];
  __syncthreads();
  const unsigned long long gen = s_gen;

  // ---- 2. segments ----------------------------------------------------------------------------
  // Groups of tpb threads, one beam per group; bpc beams per CTA and pass.
  int bpc = 1;
  while (bpc < 32 && bpc * (int)gridDim.x < cap) bpc <<= 1;
  const int tpb = kTourThreads / bpc;
  const int grp = tid / tpb, gt = tid % tpb;
  constexpr int R = 4;  // table entries per thread per chunk
  const int chunk = tpb * R;
  for (int base = blockIdx.x * bpc; base < cap; base += gridDim.x * bpc) {
    const int b = base + grp;
    const bool live = b < cap && v.active[b] != 0;
    const int nfull = live ? v.seq_len[b] / v.P : 0;
    const int* tb = v.tables + (size_t)(live ? b : 0) * v.max_pages;
    if (gt == 0) {
      s_low[grp] = nfull;      // first index with fewer than group_min sharers (or the end)
      s_cap[grp] = 0x7fffffff;  // index of the 17th segment start, if any
      s_nst[grp] = 0;
      s_carry_g[grp] = -1;      // sharer count of the entry before the chunk
    }
    __syncthreads();
    for (int c0 = 0;; c0 += chunk) {
      const bool more = c0 < s_low[grp] && c0 < s_cap[grp];
      if (!__syncthreads_or(more)) break;
      int pg[R], g[R];
      const int i0 = c0 + gt * R;
#pragma unroll
      for (int r = 0; r < R; ++r) pg[r] = (more && i0 + r < nfull) ? tb[i0 + r] : -1;
#pragma unroll
      for (int r = 0; r < R; ++r) g[r] = (pg[r] >= 0 && pg[r] < v.num_pages) ? v.refcnt[pg[r]] : 0;
      int lowl = 0x7fffffff;
#pragma unroll
      for (int r = R - 1; r >= 0; --r)
        if (more && i0 + r < nfull && g[r] < v.group_min) lowl = i0 + r;
      if (lowl != 0x7fffffff) atomicMin(&s_low[grp], lowl);
      s_pref[tid] = g[R - 1];  // the sharer count before the next thread's first entry
      __syncthreads();
      const int lim = min(s_low[grp], s_cap[grp]);
      const int gprev0 = gt > 0 ? s_pref[tid - 1] : s_carry_g[grp];
      const int carry_g = s_pref[grp * tpb + tpb - 1];
      int nst = 0, gp = gprev0;
#pragma unroll
      for (int r = 0; r < R; ++r) {
        if (more && i0 + r < lim && g[r] != gp) ++nst;
        gp = g[r];
      }
      __syncthreads();  // s_pref is reused by the scan
      int gtotal;
      int d = s_nst[grp] + group_exclusive_scan(nst, tpb, tmp, s_pref, &gtotal);
      gp = gprev0;
#pragma unroll
      for (int r = 0; r < R; ++r) {
        if (more && i0 + r < lim && g[r] != gp) {
          if (d < kMaxSegDepth) {
            s_start[grp][d] = i0 + r;
            s_spage[grp][d] = pg[r];
          } else if (d == kMaxSegDepth) {
            s_cap[grp] = i0 + r;  // deeper levels stay on the per-beam path
          }
          ++d;
        }
        gp = g[r];
      }
      __syncthreads();
      if (gt == 0) {
        s_nst[grp] += gtotal;
        s_carry_g[grp] = carry_g;
      }
      __syncthreads();
    }
    const int cover = min(s_low[grp], s_cap[grp]);
    const int nseg = min(s_nst[grp], kMaxSegDepth);
    if (live && gt < nseg) {
      const int k = gt;
      const int i0 = s_start[grp][k];
      const int end = k + 1 < nseg ? s_start[grp][k + 1] : cover;
      const int p0 = s_spage[grp][k];
      const int g = v.refcnt[p0];
      // Claim the segment (the first member to get here) or wait for its id: the claim word
      // of the start page holds (generation << 32) | (id + 1), with 0 in the low word while
      // the claimer has not published yet; one atomicMax tells a member which it is.
      unsigned long long* word = v.seg_owner + p0;
      unsigned long long cur = atomicMax(word, gen << 32);
      const bool winner = (cur >> 32) != gen;
      int id;
      if (winner) {
        // One 64-bit atomic hands out the segment id (high word; < max_beams x kMaxSegDepth / 2,
        // as a segment has >= 2 members) and the offset of its member list (low word).
        const unsigned long long got = atomicAdd(reinterpret_cast<unsigned long long*>(v.ctl + kCtlSegAlloc),
                                                 (1ull << 32) | (unsigned long long)(unsigned)g);
        id = (int)(got >> 32);
        const int toks = (end - i0) * v.P;
        const int tiles = (g * v.G + 127) / 128;
        v.seg_i0[id] = i0;
        v.seg_len[id] = end - i0;
        v.seg_rep[id] = b;
        v.seg_g[id] = g;
        v.seg_mem_off[id] = (int)(got & 0xffffffffull);
        v.seg_fill[id] = 0;
        atomicAdd(&s_rowtok, g * v.G * toks);
        atomicAdd(&s_tiletok, tiles * toks);
        atomicAdd(&s_segtok, toks);
        fence_acq_rel_gpu();  // the segment's fields before its id
        atomicMax(word, (gen << 32) | (unsigned long long)(unsigned)(id + 1));
      } else {
        const uint64_t t0 = globaltimer_ns();
        for (unsigned it = 1; (cur & 0xffffffffull) == 0; ++it) {
          cur = *reinterpret_cast<volatile unsigned long long*>(word);
          if ((it & 63) == 0 && globaltimer_ns() - t0 > kWaitLimitNs) {
            set_status(v.ctl, GB_ERR_TIMEOUT);
            break;
          }
        }
        id = (int)(cur & 0xffffffffull) - 1;
        fence_acq_rel_gpu();
      }
      if (id >= 0 && id < cap * kMaxSegDepth) {
        const int slot = atomicAdd(&v.seg_fill[id], 1);
        if (slot < v.seg_g[id] && v.seg_mem_off[id] + slot < cap * kMaxSegDepth)
          v.seg_members[v.seg_mem_off[id] + slot] = b * kMaxSegDepth + k;
        v.seg_bid[b * kMaxSegDepth + k] = id;
      }
    }
    if (live && gt == 0) {
      v.seg_cover[b] = cover;
      v.seg_nseg[b] = nseg;
    } else if (!live && b < cap && gt == 0) {
      v.seg_cover[b] = 0;
      v.seg_nseg[b] = 0;
    }
    __syncthreads();
  }
  if (tid == 0 && s_segtok > 0) {
    atomicAdd(&v.ctl[kCtlSegRowTok], s_rowtok);
    atomicAdd(&v.ctl[kCtlSegTileTok], s_tiletok);
    atomicAdd(&v.ctl[kCtlSegTok], s_segtok);
  }
  if (!grid_sync(v, &s_fail)) return;

  // ---- 3. work list, part 1: split and unit-length histogram ---------------------------------------
  // Each segment has ceil(g G / 128) query tiles; each tile is split along the segment's
  // tokens into pieces of `split` tokens (a multiple of the grouped kernel's 128-token K/V
  // tile) so that the list has about two units per multiprocessor and no beam needs more
  // than kMaxSegRecords partial records.
  const int nseg_all = v.ctl[kCtlSegAlloc + 1];  // the high word of the little-endian pair
  if (blockIdx.x == 0 && tid == 0) {
    v.ctl[kCtlSegCount] = nseg_all;
    v.ctl[kCtlSegMembers] = v.ctl[kCtlSegAlloc];
  }
  if (tid == 0) {
    const long long work = (long long)v.ctl[kCtlSegTileTok] * v.Hkv;  // tile-tokens over all heads
    const long long target_units = (long long)GB_SEG_UNITS_PCT * (v.num_sms > 0 ? v.num_sms : 1) / 100;
    int split = (int)(((work + target_units - 1) / target_units + 127) / 128 * 128);
    const int max_tokens = v.max_pages * v.P;
    const int min_split =
        ((max_tokens + (kMaxSegRecords - kMaxSegDepth) - 1) / (kMaxSegRecords - kMaxSegDepth) + 127) / 128 * 128;
    s_split = max(split, max(128, min_split));
  }
  __syncthreads();
  const int split = s_split;
  const int full_len = min(split / 128, kSegLenBuckets - 1);
  int* g_hist = v.seg_hist;                   // unit counts per length bucket
  int* g_fill = v.seg_hist + kSegLenBuckets;  // units placed so far per bucket
  for (int s = blockIdx.x * blockDim.x + tid; s < nseg_all; s += gridDim.x * blockDim.x) {
    const int tiles = (v.seg_g[s] * v.G + 127) / 128;
    const int toks = v.seg_len[s] * v.P;
    const int splits = (toks + split - 1) / split;
    v.seg_splits[s] = splits;
    const int last_len = min((toks - (splits - 1) * split + 127) / 128, kSegLenBuckets - 1);
    if (splits > 1) atomicAdd(&g_hist[full_len], tiles * (splits - 1));
    atomicAdd(&g_hist[last_len], tiles);
  }
  if (!grid_sync(v, &s_fail)) return;

  // ---- 4. work list, part 2: longest units first, and the beams' record offsets -------------------
  {
    // Units of bucket kSegLenBuckets - 1 - t first: an exclusive scan in that (longest-first) order.
    const int bk = kSegLenBuckets - 1 - tid;
    const int c = tid < kSegLenBuckets ? g_hist[bk] : 0;
    int sum;
    const int pre = block_exclusive_scan(c, tmp, &sum);
    if (tid < kSegLenBuckets) s_hist[bk] = pre;
    if (tid == 0) s_total = sum;
    __syncthreads();
  }
  const int total = s_total;
  const int wcap = cap * kMaxSegRecords;
  for (int s = blockIdx.x * blockDim.x + tid; s < nseg_all; s += gridDim.x * blockDim.x) {
    const int tiles = (v.seg_g[s] * v.G + 127) / 128;
    const int toks = v.seg_len[s] * v.P;
    const int splits = v.seg_splits[s];
    for (int sp = 0; sp < splits; ++sp) {
      const int len = min((min(toks - sp * split, split) + 127) / 128, kSegLenBuckets - 1);
      const int e0 = s_hist[len] + atomicAdd(&g_fill[len], tiles);
      for (int t = 0; t < tiles; ++t) {
        const int e = e0 + t;
        if (e < wcap) {
          v.seg_tile_seg[e] = s;
          v.seg_tile_t[e] = t;
          v.seg_tile_split[e] = sp;
        }
      }
    }
  }
  // The list holds at most 9 * max_beams + 2 * SMs entries (each beam sits in at most
  // kMaxSegDepth segments of >= 2 sharers) and a beam at most kMaxSegDepth + 32 records,
  // so neither limit is reached for pools of 8 beams or more.  Should the list still
  // overflow, the step is left entirely to the per-beam path.
  const bool overflow = total > wcap;
  // Record offsets: one lane per (beam, depth), 16 lanes per beam, an exclusive scan of the
  // segments' splits along the depths.
  static_assert(kMaxSegDepth == 16, "16 lanes per beam");
  for (int e = blockIdx.x * blockDim.x + tid; e < ((cap * kMaxSegDepth + 31) & ~31);
       e += gridDim.x * blockDim.x) {
    const int b = e / kMaxSegDepth, k = e % kMaxSegDepth;
    const int ns = b < cap ? v.seg_nseg[b] : 0;
    const int n = k < ns ? v.seg_splits[v.seg_bid[e]] : 0;
    int inc = n;
#pragma unroll
    for (int o = 1; o < kMaxSegDepth; o <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, inc, o, kMaxSegDepth);
      if (k >= o) inc += y;
    }
    const int off = __shfl_sync(0xffffffffu, inc, kMaxSegDepth - 1, kMaxSegDepth);  // the beam's records
    if (k < ns) v.seg_rec_off[e] = inc - n;
    if (b < cap && k == 0) {
      const bool drop = overflow || off > kMaxSegRecords;
      if (drop) {
        v.seg_cover[b] = 0;
        v.seg_nseg[b] = 0;
      }
      v.seg_nrec[b] = drop ? 0 : off;
    }
  }
  if (blockIdx.x == 0 && tid == 0) {
    v.ctl[kCtlSegSplit] = split;
    v.ctl[kCtlSegTiles] = overflow ? 0 : total;
  }
  pdl_launch_dependents();
}

// Grid of one CTA per SM at most (every CTA resident, which the grid barriers need).
// The active slot the tournament would rank last (Algorithm 1's eviction under KV saturation
// takes the trace with the lowest running mean, Section 3.2): the largest (rank key, slot)
// pair, i.e. NaN means first, then the lowest mean, ties to the higher slot.  One CTA.
__global__ void __launch_bounds__(1024) k_last_ranked(PoolView v, int* __restrict__ slot_out) {
  pdl_wait();
  pdl_launch_dependents();
  __shared__ unsigned long long s_best[32];
  unsigned long long best = 0;  // below every real key: (rank key << 32 | slot) + 1
  for (int s = threadIdx.x; s < v.max_beams; s += blockDim.x)
    if (v.active[s]) {
      const unsigned long long key = (((unsigned long long)rank_key(v.mean[s]) << 32) | (unsigned)s) + 1;
      best = key > best ? key : best;
    }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const unsigned long long y = __shfl_xor_sync(0xffffffffu, best, o);
    best = y > best ? y : best;
  }
  if ((threadIdx.x & 31) == 0) s_best[threadIdx.x >> 5] = best;
  __syncthreads();
  if (threadIdx.x < 32) {
    best = threadIdx.x < (int)(blockDim.x >> 5) ? s_best[threadIdx.x] : 0;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const unsigned long long y = __shfl_xor_sync(0xffffffffu, best, o);
      best = y > best ? y : best;
    }
    if (threadIdx.x == 0) *slot_out = best == 0 ? -1 : (int)((best - 1) & 0xffffffffull);
  }
}

// About four beams per CTA in the segment phase (a parent per CTA or fewer in the fork), and
// never more CTAs than SMs: every barrier's cost grows with the CTAs that meet at it.
static int tournament_grid(const gb_pool* pool) {
  const int beams = pool->view.max_beams;
  int g = pool->view.grouped ? (beams + 3) / 4 : beams;
  if (g > pool->num_sms) g = pool->num_sms;
  return g < 1 ? 1 : g;
}

cudaError_t launch_prune_branch(gb_pool* pool, int K, int fanout, int warmup, const uint8_t* elig,
                                int32_t* parent_out, uint8_t* pruned_out, uint32_t* lineage_out, cudaStream_t s) {
  TourArgs a{};
  a.prune = 1;
  a.C = pool->capacity > 0 ? pool->capacity : pool->view.max_beams;
  a.K = K;
  a.fanout = fanout;
  a.warmup = warmup;
  a.elig = elig;
  a.parent_out = parent_out;
  a.pruned_out = pruned_out;
  a.lineage_out = reinterpret_cast<unsigned*>(lineage_out);
  pool->launches += 1;
  return launch_pdl(k_tournament, tournament_grid(pool), kTourThreads, 0, s, pool->view, a);
}

cudaError_t rebuild_segments(gb_pool* pool, cudaStream_t s) {
  if (!pool->view.grouped) return cudaSuccess;
  TourArgs a{};
  a.prune = 0;
  pool->launches += 1;
  return launch_pdl(k_tournament, tournament_grid(pool), kTourThreads, 0, s, pool->view, a);
}

}  // namespace gb

using namespace gb;

extern "C" gb_status gb_pool_last_ranked(gb_pool* pool, int32_t* slot_out_dev, gb_stream_t stream) {
  if (!pool || !slot_out_dev) return GB_ERR_INVALID;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  launch_pdl(k_last_ranked, 1, 1024, 0, s, pool->view, slot_out_dev);
  pool->launches += 1;
  return check_launch(pool, "last_ranked");
}
