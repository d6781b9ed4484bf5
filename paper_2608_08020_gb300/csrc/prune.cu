// One tournament round (Algorithm 1, Tournament; Eq. 2 and Eq. 3) as a single
// launch.  Every CTA ranks the active slots redundantly (bitonic sort of
// 64-bit keys in shared memory) and derives the same routing; the children
// are then spread over the CTAs, each forking its children's block tables
// with net refcount updates; the last CTA to finish writes the per-slot
// metadata and outputs.
//
// Why no page is freed too early: a page referenced by a surviving beam keeps
// that reference for the whole round (survivors are never pruned), so only
// pages referenced by pruned beams alone can reach zero, and no child ever
// takes a reference to such a page.  A decrement that returns 1 therefore
// frees the page for good.
#include "internal.cuh"

namespace gb {

// Unsigned key whose ascending order is: larger mean first, +0 == -0, NaN last.
__device__ __forceinline__ unsigned rank_key(float m) {
  if (isnan(m)) return 0xffffffffu;
  if (m == 0.f) m = 0.f;
  const unsigned u = __float_as_uint(m);
  const unsigned asc = (u & 0x80000000u) ? ~u : (u | 0x80000000u);
  return ~asc;
}

__global__ void __launch_bounds__(1024) k_prune_branch(PoolView v, int C, int K, int fanout, int warmup,
                                                        const uint8_t* __restrict__ elig_mask,
                                                        int* __restrict__ parent_out,
                                                        uint8_t* __restrict__ pruned_out,
                                                        unsigned* __restrict__ lineage_out) {
  pdl_wait();
  pdl_launch_dependents();
  __shared__ unsigned long long keys[kMaxBeams];
  __shared__ int ord[kMaxBeams];     // rank -> slot
  __shared__ int blist[kMaxBeams];   // eligible parents in rank order
  __shared__ int cslot[kMaxBeams];   // child k -> slot
  __shared__ int cpar[kMaxBeams];    // child k -> parent slot
  __shared__ int childof[kMaxBeams]; // slot -> child index or -1
  __shared__ unsigned char s_act[kMaxBeams], s_elig[kMaxBeams], s_pruned[kMaxBeams];
  __shared__ int tmp[33];
  __shared__ int s_nchild, s_last;
  const int tid = threadIdx.x;
  const int cap = v.max_beams;  // physical slots; C <= cap is the tree's capacity

  // 1. Active slots, eligibility, compaction into sort keys.
  const bool act = tid < cap && v.active[tid] != 0;
  const bool elig = act && v.gen[tid] >= warmup && (elig_mask == nullptr || elig_mask[tid] != 0);
  if (tid < kMaxBeams) {
    s_act[tid] = act;
    s_elig[tid] = elig;
    s_pruned[tid] = 0;
    childof[tid] = -1;
  }
  int N;
  const int pos = block_exclusive_scan(act ? 1 : 0, tmp, &N);
  int npow = 1;
  while (npow < N) npow <<= 1;
  if (tid < npow) keys[tid] = ~0ull;
  __syncthreads();
  if (act) keys[pos] = ((unsigned long long)rank_key(v.mean[tid]) << 32) | (unsigned)tid;
  __syncthreads();
  // 2. Bitonic sort, ascending.
  for (int k = 2; k <= npow; k <<= 1) {
    for (int j = k >> 1; j > 0; j >>= 1) {
      const int ixj = tid ^ j;
      if (tid < npow && ixj > tid) {
        const unsigned long long a = keys[tid], b = keys[ixj];
        const bool asc = (tid & k) == 0;
        if ((a > b) == asc) {
          keys[tid] = b;
          keys[ixj] = a;
        }
      }
      __syncthreads();
    }
  }
  if (tid < N) ord[tid] = (int)(keys[tid] & 0xffffffffu);
  __syncthreads();

  // 3. Routing (identical in every CTA).
  int nchild = 0;
  if (N > 0 && N < C) {
    // Case 1 (Eq. 2): top min(C - N, |B|) eligible traces, one child each, into vacant slots.
    const bool f = tid < N && s_elig[ord[tid]];
    int nb;
    const int pb = block_exclusive_scan(f ? 1 : 0, tmp, &nb);
    if (f) blist[pb] = ord[tid];
    nchild = min(C - N, nb);
    const bool vac = tid < cap && !act;
    int nv;
    const int pv = block_exclusive_scan(vac ? 1 : 0, tmp, &nv);
    if (vac && pv < nchild) cslot[pv] = tid;
    __syncthreads();
    if (tid < nchild) cpar[tid] = blist[tid];
  } else if (N > 0) {
    // Case 2 (Eq. 3, fan-out f; N = C): prune the bottom K_eff, branch the top eligible survivors.
    const int Kc = K < 0 ? 0 : (K > N ? N : K);
    const int nsurv = N - Kc;
    const bool f = tid < nsurv && s_elig[ord[tid]];
    int nb;
    const int pb = block_exclusive_scan(f ? 1 : 0, tmp, &nb);
    if (f) blist[pb] = ord[tid];
    const long long cap_children = (long long)(fanout - 1) * nb;
    nchild = (int)(Kc < cap_children ? Kc : cap_children);
    if (tid >= N - nchild && tid < N) s_pruned[ord[tid]] = 1;
    __syncthreads();
    const bool pr = tid < cap && s_pruned[tid];
    int np;
    const int pp = block_exclusive_scan(pr ? 1 : 0, tmp, &np);
    if (pr) cslot[pp] = tid;
    __syncthreads();
    if (tid < nchild) cpar[tid] = blist[tid / (fanout - 1)];
  }
  __syncthreads();
  if (tid < nchild) childof[cslot[tid]] = tid;
  if (tid == 0) s_nchild = nchild;
  __syncthreads();

  // 4. Fork block tables: child k in slot s takes parent p's table.
  for (int k = blockIdx.x; k < nchild; k += gridDim.x) {
    const int s = cslot[k], p = cpar[k];
    const int old_n = s_act[s] ? (v.seq_len[s] + v.P - 1) / v.P : 0;
    const int new_n = (v.seq_len[p] + v.P - 1) / v.P;
    const int m = old_n > new_n ? old_n : new_n;
    int* ts = v.tables + (size_t)s * v.max_pages;
    const int* tp = v.tables + (size_t)p * v.max_pages;
    for (int i = tid; i < m; i += blockDim.x) {
      const int old = i < old_n ? ts[i] : -1;
      const int nw = i < new_n ? tp[i] : -1;
      if (old == nw) continue;
      if (nw >= 0) atomicAdd(&v.refcnt[nw], 1);
      if (old >= 0) unref_page(v, old);
      if (i < new_n) ts[i] = nw;
    }
  }

  // 5. The last CTA writes metadata and outputs.
  __threadfence();
  __syncthreads();
  if (tid == 0) s_last = atomicAdd(&v.ctl[kCtlDone], 1) == (int)gridDim.x - 1;
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  const unsigned lin0 = (unsigned)v.ctl[kCtlNextLineage];
  if (tid < s_nchild) {
    const int s = cslot[tid], p = cpar[tid];
    v.seq_len[s] = v.seq_len[p];
    v.mean[s] = v.mean[p];
    v.nsteps[s] = v.nsteps[p];
    v.gen[s] = 0;
    v.active[s] = 1;
    v.lineage[s] = lin0 + tid;
  }
  if (tid < cap) {
    const int k = childof[tid];
    if (parent_out) parent_out[tid] = k >= 0 ? cpar[k] : (s_act[tid] ? tid : -1);
    if (pruned_out) pruned_out[tid] = s_pruned[tid];
    if (lineage_out) lineage_out[tid] = k >= 0 ? lin0 + k : v.lineage[tid];
  }
  if (tid == 0) {
    v.ctl[kCtlNextLineage] = (int)(lin0 + s_nchild);
    v.ctl[kCtlDone] = 0;
  }
}

// Apply a tournament decided elsewhere (another pool's parent_out): every slot s with
// parent_of[s] >= 0 and != s becomes a child of parent_of[s] - its old references go, it
// takes the parent's table (+1 on every page), length, mean and count, gen = 0 and a new
// lineage id, in ascending slot order.  One CTA, one warp per child (lanes over table
// entries): reference counts change by atomics, so the end state does not depend on the
// order; the parents must not be children themselves (survivors keep parent_of[p] = p).
__global__ void __launch_bounds__(1024) k_fork_slots(PoolView v, const int* __restrict__ parent_of) {
  pdl_wait();
  pdl_launch_dependents();
  __shared__ int cslot[kMaxBeams], cpar[kMaxBeams];
  __shared__ int tmp[33];
  const int tid = threadIdx.x;
  const int p = tid < v.max_beams ? parent_of[tid] : -1;
  const bool child = tid < v.max_beams && p >= 0 && p < v.max_beams && p != tid;
  if (tid < v.max_beams && p >= v.max_beams) set_status(v.ctl, GB_ERR_INVALID);
  int nchild;
  const int k = block_exclusive_scan(child ? 1 : 0, tmp, &nchild);
  if (child) {
    cslot[k] = tid;
    cpar[k] = p;
  }
  __syncthreads();
  const int lane = tid & 31, nwarps = blockDim.x >> 5;
  for (int c = tid >> 5; c < nchild; c += nwarps) {
    const int s = cslot[c], par = cpar[c];
    const int old_n = v.active[s] ? (v.seq_len[s] + v.P - 1) / v.P : 0;
    const int new_n = (v.seq_len[par] + v.P - 1) / v.P;
    const int m = old_n > new_n ? old_n : new_n;
    int* ts = v.tables + (size_t)s * v.max_pages;
    const int* tp = v.tables + (size_t)par * v.max_pages;
    for (int i = lane; i < m; i += 32) {
      const int old = i < old_n ? ts[i] : -1;
      const int nw = i < new_n ? tp[i] : -1;
      if (old == nw) continue;
      if (nw >= 0) atomicAdd(&v.refcnt[nw], 1);
      if (old >= 0) unref_page(v, old);
      if (i < new_n) ts[i] = nw;
    }
  }
  __syncthreads();
  const unsigned lin0 = (unsigned)v.ctl[kCtlNextLineage];
  if (tid < nchild) {
    const int s = cslot[tid], par = cpar[tid];
    v.seq_len[s] = v.seq_len[par];
    v.mean[s] = v.mean[par];
    v.nsteps[s] = v.nsteps[par];
    v.gen[s] = 0;
    v.active[s] = 1;
    v.lineage[s] = lin0 + tid;
  }
  if (tid == 0) v.ctl[kCtlNextLineage] = (int)(lin0 + nchild);
}

cudaError_t launch_prune_branch(gb_pool* pool, int K, int fanout, int warmup, const uint8_t* elig,
                                int32_t* parent_out, uint8_t* pruned_out, uint32_t* lineage_out, cudaStream_t s) {
  const int grid = pool->view.max_beams < pool->num_sms ? pool->view.max_beams : pool->num_sms;
  const int C = pool->capacity > 0 ? pool->capacity : pool->view.max_beams;
  const cudaError_t e = launch_pdl(k_prune_branch, grid, 1024, 0, s, pool->view, C, K, fanout, warmup, elig,
                                   parent_out, pruned_out, reinterpret_cast<unsigned*>(lineage_out));
  pool->launches += 1;
  return e;
}

}  // namespace gb

using namespace gb;

extern "C" gb_status gb_fork_slots(gb_pool* pool, const int32_t* parent_of_dev, gb_stream_t stream) {
  if (!pool || !parent_of_dev) return GB_ERR_INVALID;
  if (!pool->seeded) return fail(pool, GB_ERR_STATE, "pool not seeded");
  if (pool->next_layer != 0) return fail(pool, GB_ERR_STATE, "fork_slots inside an open step");
  if (pool->cfg.max_beams > kMaxBeams) return fail(pool, GB_ERR_UNSUPPORTED, "fork_slots: too many slots");
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  prof_begin(pool, GB_PROF_PRUNE, s);
  launch_pdl(k_fork_slots, 1, 1024, 0, s, pool->view, parent_of_dev);
  pool->launches += 1;
  gb_status st = check_launch(pool, "fork_slots");
  if (st != GB_OK) return st;
  if (rebuild_segments(pool, s) != cudaSuccess) return check_launch(pool, "segments");
  prof_end(pool, GB_PROF_PRUNE, s);
  return GB_OK;
}

extern "C" gb_status gb_pool_set_capacity(gb_pool* pool, int capacity) {
  if (!pool) return GB_ERR_INVALID;
  if (capacity < 1 || capacity > pool->cfg.max_beams)
    return fail(pool, GB_ERR_INVALID, "set_capacity: 1 <= capacity <= max_beams required");
  pool->capacity = capacity;
  return GB_OK;
}

extern "C" gb_status gb_prune_branch(gb_pool* pool, int K, int fanout, int warmup, const uint8_t* eligible_dev,
                                     int32_t* parent_out_dev, uint8_t* pruned_out_dev, uint32_t* lineage_out_dev,
                                     gb_stream_t stream) {
  if (!pool) return GB_ERR_INVALID;
  if (K < 0 || fanout < 2) return fail(pool, GB_ERR_INVALID, "prune_branch: K >= 0 and fanout >= 2 required");
  if (!pool->seeded) return fail(pool, GB_ERR_STATE, "pool not seeded");
  if (pool->next_layer != 0) return fail(pool, GB_ERR_STATE, "prune_branch inside an open step");
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  prof_begin(pool, GB_PROF_PRUNE, s);
  launch_prune_branch(pool, K, fanout, warmup, eligible_dev, parent_out_dev, pruned_out_dev, lineage_out_dev, s);
  gb_status st = check_launch(pool, "prune_branch");
  if (st != GB_OK) return st;
  if (rebuild_segments(pool, s) != cudaSuccess) return check_launch(pool, "segments");
  prof_end(pool, GB_PROF_PRUNE, s);
  return GB_OK;
}
