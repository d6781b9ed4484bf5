// The log-sum-exp merge of a layer-step's partial attention records, run at the end of the
// attention launch itself (k_attention, k_decode_mma) rather than as a launch of its own.
//
// Each (beam b, KV head h) pair has R = npb + nseg records: npb split-KV records of the
// per-beam warps whose chunk range meets the pair's chunks (warp w's record of the pair is
// number w + b * Hkv + h), and, on the grouped path, nseg records of the beam's shared-prefix
// segments.  A per-beam warp counts each record it writes in pair_cnt[b * Hkv + h] (release:
// fence, then the add); a grouped CTA counts itself in ctl[kCtlGrpDone] once all of its
// records are written.  After their own work, the merging CTAs (the launch's caller names
// them: cta of nctas) take the pairs p = cta + nctas * (warp + k * warps per CTA); a warp waits
// (bounded) until pair_cnt[p] == npb and, when nseg > 0, every grouped CTA has finished, then
// merges the R records into out[b][h * G + g][:]: running max M of the records' m,
// acc = sum o * 2^(m - M), L = sum l * 2^(m - M), out = acc / L.
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

// Merge the records of pair (b, h) into out[b][h * G + g][:] (one warp; lane l owns the
// elements 4l .. 4l + 3 of every head g).  The records exist: the caller waited for them.
template <int G>
__device__ __forceinline__ void merge_pair(const PoolView& v, int b, int h, int first, int npb, int nseg,
                                           float* __restrict__ out) {
  constexpr int D = 128, GD = G * D;
  constexpr int RB = G >= 8 ? 1 : 16 / G;  // records per batch of loads: 8-16 float4 in flight per lane
  const int lane = threadIdx.x & 31;
  const size_t rf = (size_t)v.record_floats, gstride = (size_t)v.Hkv * rf;
  const int bh = b * v.Hkv + h, R = npb + nseg;
  const float* prec = v.partials + (size_t)(first + bh) * rf;
  const float* grec = v.grec + ((size_t)b * kMaxSegRecords * v.Hkv + h) * rf;
  float M[G], L[G];
  float4 acc[G];
#pragma unroll
  for (int g = 0; g < G; ++g) {
    M[g] = -INFINITY;
    L[g] = 0.f;
    acc[g] = make_float4(0.f, 0.f, 0.f, 0.f);
  }
  for (int r0 = 0; r0 < R; r0 += RB) {
    float4 x[RB][G];
    float mk[RB][G], lk[RB][G];
#pragma unroll
    for (int k = 0; k < RB; ++k) {
      const int r = r0 + k;
      if (r < R) {
        // L2 loads: the records were written by other SMs during this launch.
        const float* rec = r < npb ? prec + (size_t)r * rf : grec + (size_t)(r - npb) * gstride;
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
      float mnew = M[g];
#pragma unroll
      for (int k = 0; k < RB; ++k) mnew = fmaxf(mnew, mk[k][g]);
      if (mnew == -INFINITY) continue;
      if (mnew > M[g]) {  // M = -inf the first time: acc and L are still 0
        const float a = M[g] == -INFINITY ? 0.f : exp2f(M[g] - mnew);
        acc[g].x *= a;
        acc[g].y *= a;
        acc[g].z *= a;
        acc[g].w *= a;
        L[g] *= a;
        M[g] = mnew;
      }
#pragma unroll
      for (int k = 0; k < RB; ++k) {
        const float sc = mk[k][g] == -INFINITY ? 0.f : exp2f(mk[k][g] - M[g]);
        acc[g].x = fmaf(x[k][g].x, sc, acc[g].x);
        acc[g].y = fmaf(x[k][g].y, sc, acc[g].y);
        acc[g].z = fmaf(x[k][g].z, sc, acc[g].z);
        acc[g].w = fmaf(x[k][g].w, sc, acc[g].w);
        L[g] = fmaf(lk[k][g], sc, L[g]);
      }
    }
  }
  float* ob = out + ((size_t)b * v.Hq + (size_t)h * G) * D;
  const bool vec_out = (reinterpret_cast<uintptr_t>(out) & 15) == 0;
#pragma unroll
  for (int g = 0; g < G; ++g) {
    const float4 res = make_float4(acc[g].x / L[g], acc[g].y / L[g], acc[g].z / L[g], acc[g].w / L[g]);
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

// The merge phase of an attention launch: `mode` selects the plan (0 per-beam, 1 with
// segments), W = warps of the per-beam role, ng = CTAs of the grouped role (0 without one),
// out = [max_beams][Hq][128] fp32.
template <int G>
__device__ __forceinline__ void combine_pairs(const PoolView& v, int mode, int W, int ng, int cta, int nctas,
                                              float* __restrict__ out) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, nw = blockDim.x >> 5;
  const int npairs = v.max_beams * v.Hkv;
  const bool ok = v.ctl[kCtlStepOk] != 0;
  const int* off = plan_off(v, mode);
  const int* nn = plan_n(v, mode);
  const int Tot = off[v.max_beams];
  const int c = Tot > 0 ? (Tot + W - 1) / W : 1;  // chunks per per-beam warp
  for (int p = cta + nctas * warp; p < npairs; p += nctas * nw) {
    const int b = p / v.Hkv, h = p - b * v.Hkv;
    const bool act = ok && v.active[b] != 0;
    const int n = act ? nn[b] : 0;
    const int nseg = (act && mode == 1 && v.grouped) ? v.seg_nrec[b] : 0;
    const int o0 = off[b] + h * n;
    const int first = o0 / c;
    const int npb = n > 0 ? (o0 + n - 1) / c - first + 1 : 0;
    if (npb + nseg > 0 && wait_pair_records(v, p, npb, nseg > 0 ? ng : 0)) {
      merge_pair<G>(v, b, h, first, npb, nseg, out);
    } else {
      if (npb + nseg > 0 && lane == 0) set_status(v.ctl, GB_ERR_TIMEOUT);  // kept if already set
      zero_pair<G>(v, b, h, out);
    }
  }
}

}  // namespace gb
