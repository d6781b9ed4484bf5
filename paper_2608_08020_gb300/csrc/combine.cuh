// The log-sum-exp merge of a layer-step's partial attention records, run at the end of the
// attention launch itself (k_attention, k_decode_mma) rather than as a launch of its own.
//
// Each (beam b, KV head h) pair has R = nseg + npb records: on the grouped path, nseg records
// of the beam's shared-prefix segments, and npb split-KV records of the per-beam warps whose
// chunk range meets the pair's chunks (warp w's record of the pair is number w + b * Hkv + h).
// A grouped CTA counts itself in ctl[kCtlGrpDone] once all of its records are written; a
// per-beam warp counts each record it writes in pair_cnt[b * Hkv + h] (release: fence, then
// the add).  After its own work, every warp of the merging CTAs takes pairs from the counter
// ctl[kCtlPairNext] until none is left, so the warps that finish first take the pairs and the
// last ones to finish find none.  Per pair it folds the segment records first (a bounded wait
// until every grouped CTA has finished, long past on a large step), then waits (bounded) until
// pair_cnt[p] == npb and folds the split-KV records, so what remains after the pair's last
// record is one batch of loads: running max M of the records' m, acc = sum o * 2^(m - M),
// L = sum l * 2^(m - M), out[b][h * G + g][:] = acc / L.
//
// The waits end because every CTA they wait on gets an SM: the callers only let CTAs merge
// that are resident together with the ones they wait on, or that wait only on CTAs which never
// wait (k_attention).  Each wait is bounded and gives up as soon as the pool's status word is
// set.  The counters are zeroed by k_append, the launch that precedes every attention launch.
#pragma once
#include <cuda_runtime.h>
#include <math.h>
#include "internal.cuh"
#include "ptx.cuh"

namespace gb {

// A per-beam warp has written the record of pair bh: make the writes visible, then count it.
__device__ __forceinline__ void record_arrive(const PoolView& v, int bh, int lane) {
  fence_acq_rel_gpu();
  __syncwarp();
  if (lane == 0) atomicAdd(&v.pair_cnt[bh], 1);
}

// A grouped CTA has written all of its records (called by every thread of the CTA).
__device__ __forceinline__ void grouped_cta_done(const PoolView& v) {
  __syncthreads();
  if (threadIdx.x == 0) {
    fence_acq_rel_gpu();
    atomicAdd(&v.ctl[kCtlGrpDone], 1);
  }
}

// Wait, with the whole warp polling, until pair p has npb split-KV records and ng grouped
// CTAs have finished.  False on a timeout or when an error status is set.
__device__ __forceinline__ bool wait_pair_records(const PoolView& v, int p, int npb, int ng) {
  const uint64_t t0 = globaltimer_ns();
  unsigned ns = 32;
  while (true) {
    const int a = npb > 0 ? ld_acquire_gpu(&v.pair_cnt[p]) : 0;
    const int g = ng > 0 ? ld_acquire_gpu(&v.ctl[kCtlGrpDone]) : 0;
    if (__all_sync(0xffffffffu, a >= npb && g >= ng)) return true;
    if (__any_sync(0xffffffffu, *reinterpret_cast<volatile int*>(&v.ctl[kCtlStatus]) != GB_OK ||
                                    globaltimer_ns() - t0 > kWaitLimitNs))
      return false;
    __nanosleep(ns);
    ns = ns < 512 ? 2 * ns : ns;
  }
}

// The running state of one pair's merge (one warp; lane l owns the elements 4l .. 4l + 3 of
// every head g of the pair).
template <int G>
struct MergeState {
  float M[G], L[G];
  float4 acc[G];
};

template <int G>
__device__ __forceinline__ void merge_init(MergeState<G>& st) {
#pragma unroll
  for (int g = 0; g < G; ++g) {
    st.M[g] = -INFINITY;
    st.L[g] = 0.f;
    st.acc[g] = make_float4(0.f, 0.f, 0.f, 0.f);
  }
}

// Fold the records rec0, rec0 + stride, ... (cnt of them) into the state.  The records exist:
// the caller waited for them.
template <int G>
__device__ __forceinline__ void merge_fold(MergeState<G>& st, const float* rec0, size_t stride, int cnt) {
  constexpr int D = 128, GD = G * D;
  constexpr int RB = G >= 8 ? 1 : 16 / G;  // records per batch of loads: 8-16 float4 in flight per lane
  const int lane = threadIdx.x & 31;
  for (int r0 = 0; r0 < cnt; r0 += RB) {
    float4 x[RB][G];
    float mk[RB][G], lk[RB][G];
#pragma unroll
    for (int k = 0; k < RB; ++k) {
      if (r0 + k < cnt) {
        // L2 loads: the records were written by other SMs during this launch.
        const float* rec = rec0 + (size_t)(r0 + k) * stride;
#pragma unroll
        for (int g = 0; g < G; ++g) {
          x[k][g] = __ldcg(reinterpret_cast<const float4*>(rec + g * D) + lane);
          mk[k][g] = __ldcg(rec + GD + g);
          lk[k][g] = __ldcg(rec + GD + G + g);
        }
      } else {
#pragma unroll
        for (int g = 0; g < G; ++g) {
          x[k][g] = make_float4(0.f, 0.f, 0.f, 0.f);
          mk[k][g] = -INFINITY;  // a record that saw no token (or none at all) adds nothing
          lk[k][g] = 0.f;
        }
      }
    }
#pragma unroll
    for (int g = 0; g < G; ++g) {
      float mnew = st.M[g];
#pragma unroll
      for (int k = 0; k < RB; ++k) mnew = fmaxf(mnew, mk[k][g]);
      if (mnew == -INFINITY) continue;
      if (mnew > st.M[g]) {  // M = -inf the first time: acc and L are still 0
        const float a = st.M[g] == -INFINITY ? 0.f : exp2f(st.M[g] - mnew);
        st.acc[g].x *= a;
        st.acc[g].y *= a;
        st.acc[g].z *= a;
        st.acc[g].w *= a;
        st.L[g] *= a;
        st.M[g] = mnew;
      }
#pragma unroll
      for (int k = 0; k < RB; ++k) {
        const float sc = mk[k][g] == -INFINITY ? 0.f : exp2f(mk[k][g] - st.M[g]);
        st.acc[g].x = fmaf(x[k][g].x, sc, st.acc[g].x);
        st.acc[g].y = fmaf(x[k][g].y, sc, st.acc[g].y);
        st.acc[g].z = fmaf(x[k][g].z, sc, st.acc[g].z);
        st.acc[g].w = fmaf(x[k][g].w, sc, st.acc[g].w);
        st.L[g] = fmaf(lk[k][g], sc, st.L[g]);
      }
    }
  }
}

// out[b][h * G + g][:] = acc / L.
template <int G>
__device__ __forceinline__ void merge_write(const PoolView& v, const MergeState<G>& st, int b, int h,
                                            float* __restrict__ out) {
  constexpr int D = 128;
  const int lane = threadIdx.x & 31;
  float* ob = out + ((size_t)b * v.Hq + (size_t)h * G) * D;
  const bool vec_out = (reinterpret_cast<uintptr_t>(out) & 15) == 0;
#pragma unroll
  for (int g = 0; g < G; ++g) {
    const float4 res = make_float4(st.acc[g].x / st.L[g], st.acc[g].y / st.L[g], st.acc[g].z / st.L[g],
                                   st.acc[g].w / st.L[g]);
    float* d = ob + g * D + 4 * lane;
    if (vec_out) {
      *reinterpret_cast<float4*>(d) = res;
    } else {
      d[0] = res.x;
      d[1] = res.y;
      d[2] = res.z;
      d[3] = res.w;
    }
  }
}

// Zero the output rows of pair (b, h) (an inactive beam, or a failed wait).
template <int G>
__device__ __forceinline__ void zero_pair(const PoolView& v, int b, int h, float* __restrict__ out) {
  float* ob = out + ((size_t)b * v.Hq + (size_t)h * G) * 128;
  for (int e = threadIdx.x & 31; e < G * 128; e += 32) ob[e] = 0.f;
}

// The merge phase of an attention launch, run by every warp of the merging CTAs after its own
// work: `mode` selects the plan (0 per-beam, 1 with segments), W = warps of the per-beam
// role, ng = CTAs of the grouped role (0 without one), out = [max_beams][Hq][128] fp32.
// `claim`: the warps take pairs from the counter ctl[kCtlPairNext] as they finish (for CTAs
// that start at different times) and fold a pair's segment records before they wait for its
// split-KV records; otherwise merging CTA `cta` of `nctas` takes the pairs
// p = cta + nctas * (warp + k * warps per CTA) and waits for all of a pair's records at once.
template <int G>
__device__ __forceinline__ void combine_pairs(const PoolView& v, int mode, int W, int ng, bool claim, int cta,
                                              int nctas, float* __restrict__ out) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
  const int npairs = v.max_beams * v.Hkv;
  const bool ok = v.ctl[kCtlStepOk] != 0;
  const int* off = plan_off(v, mode);
  const int* nn = plan_n(v, mode);
  const int Tot = off[v.max_beams];
  const int c = Tot > 0 ? (Tot + W - 1) / W : 1;  // chunks per per-beam warp
  const size_t rf = (size_t)v.record_floats;
  for (int k = 0;; ++k) {
    int p = cta + nctas * (warp + k * nw);
    if (claim) {
      if (lane == 0) p = atomicAdd(&v.ctl[kCtlPairNext], 1);
      p = __shfl_sync(0xffffffffu, p, 0);
    }
    if (p >= npairs) break;
    const int b = p / v.Hkv, h = p - b * v.Hkv;
    const bool act = ok && v.active[b] != 0;
    const int n = act ? nn[b] : 0;
    const int nseg = (act && mode == 1 && v.grouped) ? v.seg_nrec[b] : 0;
    const int o0 = off[b] + h * n;
    const int first = o0 / c;
    const int npb = n > 0 ? (o0 + n - 1) / c - first + 1 : 0;
    if (npb + nseg == 0) {
      zero_pair<G>(v, b, h, out);
      continue;
    }
    const float* grec = v.grec + ((size_t)b * kMaxSegRecords * v.Hkv + h) * rf;  // [b][record][Hkv]
    const float* prec = v.partials + (size_t)(first + p) * rf;                     // first + p, ...
    MergeState<G> st;
    merge_init(st);
    bool good;
    if (claim) {
      good = nseg == 0 || wait_pair_records(v, p, 0, ng);
      if (good && nseg > 0) merge_fold(st, grec, (size_t)v.Hkv * rf, nseg);
      good = good && (npb == 0 || wait_pair_records(v, p, npb, 0));
      if (good && npb > 0) merge_fold(st, prec, rf, npb);
    } else {
      good = wait_pair_records(v, p, npb, nseg > 0 ? ng : 0);
      if (good) {
        merge_fold(st, prec, rf, npb);
        merge_fold(st, grec, (size_t)v.Hkv * rf, nseg);
      }
    }
    if (good) {
      merge_write(v, st, b, h, out);
    } else {
      if (lane == 0) set_status(v.ctl, GB_ERR_TIMEOUT);  // kept if already set
      zero_pair<G>(v, b, h, out);
    }
  }
}

}  // namespace gb
