// The tournament's entry points (the kernel is in tournament.cu), the capacity of the
// tree, and gb_fork_slots: a tournament decided on another pool applied to this one.
#include "internal.cuh"

namespace gb {

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
  if (tid == 0) {
    v.ctl[kCtlNextLineage] = (int)(lin0 + nchild);
    if (nchild > 0) v.ctl[kCtlTailShared] = 1;  // children share their parents' partial tail pages
  }
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
  // One launch: the round and the shared-prefix segment rebuild that follows it.
  launch_prune_branch(pool, K, fanout, warmup, eligible_dev, parent_out_dev, pruned_out_dev, lineage_out_dev, s);
  gb_status st = check_launch(pool, "prune_branch");
  if (st != GB_OK) return st;
  prof_end(pool, GB_PROF_PRUNE, s);
  return GB_OK;
}
