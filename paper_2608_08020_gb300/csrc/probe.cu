// Scorer probe f(h) = sigmoid(w.h + b) fused with the running-mean update of
// Algorithm 1 ("s_bar <- s_bar + (f(h_n) - s_bar)/n").  One CTA of 128 threads per slot:
// 16-byte loads of the hidden row (all in flight at once for H = 4096), fp32 accumulation,
// shuffle and shared-memory reduction.
// The mean update rounds subtract, divide and add separately, in that order.
#include "internal.cuh"

namespace gb {

constexpr int kProbeThreads = 128;  // one CTA per slot

// Partial dot product of this thread's share of a hidden row with w: 16-byte loads, four
// independent iterations unrolled so that their loads are in flight together.
template <int HT>
__device__ __forceinline__ float dot_part(const void* hrow, const float* __restrict__ w, int H, int t) {
  float acc0 = 0.f, acc1 = 0.f;
  if constexpr (HT == GB_BF16) {
    const uint4* h4 = static_cast<const uint4*>(hrow);
#pragma unroll 4
    for (int e = t; e < H / 8; e += kProbeThreads) {
      const uint4 u = h4[e];
      const float4 wa = reinterpret_cast<const float4*>(w)[2 * e];
      const float4 wb = reinterpret_cast<const float4*>(w)[2 * e + 1];
      acc0 = fmaf(__uint_as_float(u.x << 16), wa.x, acc0);
      acc1 = fmaf(__uint_as_float(u.x & 0xffff0000u), wa.y, acc1);
      acc0 = fmaf(__uint_as_float(u.y << 16), wa.z, acc0);
      acc1 = fmaf(__uint_as_float(u.y & 0xffff0000u), wa.w, acc1);
      acc0 = fmaf(__uint_as_float(u.z << 16), wb.x, acc0);
      acc1 = fmaf(__uint_as_float(u.z & 0xffff0000u), wb.y, acc1);
      acc0 = fmaf(__uint_as_float(u.w << 16), wb.z, acc0);
      acc1 = fmaf(__uint_as_float(u.w & 0xffff0000u), wb.w, acc1);
    }
  } else {
    const float4* h4 = static_cast<const float4*>(hrow);
#pragma unroll 4
    for (int e = t; e < H / 4; e += kProbeThreads) {
      const float4 u = h4[e];
      const float4 wa = reinterpret_cast<const float4*>(w)[e];
      acc0 = fmaf(u.x, wa.x, acc0);
      acc1 = fmaf(u.y, wa.y, acc1);
      acc0 = fmaf(u.z, wa.z, acc0);
      acc1 = fmaf(u.w, wa.w, acc1);
    }
  }
  return acc0 + acc1;
}

template <int HT>
__global__ void __launch_bounds__(kProbeThreads) k_probe(PoolView v, const void* __restrict__ hidden, int H,
                                                         const float* __restrict__ w, float bias,
                                                         const uint8_t* __restrict__ mask, float* __restrict__ score_out,
                                                         const float* __restrict__ scores_in) {
  pdl_wait();
  pdl_launch_dependents();
  __shared__ float s_part[kProbeThreads / 32];
  const int b = blockIdx.x, t = threadIdx.x, lane = t & 31;
  if (!v.active[b]) {
    if (score_out && t == 0) score_out[b] = 0.f;
    return;
  }
  float x;
  if (scores_in) {
    x = scores_in[b];
  } else {
    const size_t es = HT == GB_BF16 ? 2 : 4;
    float acc = dot_part<HT>(static_cast<const char*>(hidden) + (size_t)b * H * es, w, H, t);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
    if (lane == 0) s_part[t >> 5] = acc;
    __syncthreads();
    float z = bias;
#pragma unroll
    for (int i = 0; i < kProbeThreads / 32; ++i) z += s_part[i];
    x = 1.0f / (1.0f + expf(-z));
    if (score_out && t == 0) score_out[b] = x;
  }
  if (t == 0 && (mask == nullptr || mask[b] != 0)) {
    const int n = v.nsteps[b] + 1;
    const float m = v.mean[b];
    const float d = __fsub_rn(x, m);
    const float q = __fdiv_rn(d, (float)n);
    v.mean[b] = __fadd_rn(m, q);
    v.nsteps[b] = n;
  }
}

cudaError_t launch_probe(gb_pool* pool, const void* hidden, int hidden_dtype, int H, const float* w, float bias,
                         const uint8_t* mask, float* score_out, const float* scores_in, cudaStream_t s) {
  const int grid = pool->view.max_beams;  // one CTA per slot
  pool->launches += 1;
  if (scores_in == nullptr) prof_begin(pool, GB_PROF_PROBE, s);
  const cudaError_t e =
      hidden_dtype == GB_BF16
          ? launch_pdl(k_probe<GB_BF16>, grid, kProbeThreads, 0, s, pool->view, hidden, H, w, bias, mask,
                       score_out, scores_in)
          : launch_pdl(k_probe<GB_F32>, grid, kProbeThreads, 0, s, pool->view, hidden, H, w, bias, mask,
                       score_out, scores_in);
  if (scores_in == nullptr) prof_end(pool, GB_PROF_PROBE, s);
  return e;
}

}  // namespace gb

using namespace gb;

extern "C" gb_status gb_score_probe(gb_pool* pool, const void* hidden_dev, int hidden_dtype, int hidden_dim,
                                    const float* w_dev, float bias, const uint8_t* boundary_mask_dev,
                                    float* score_out_dev, gb_stream_t stream) {
  if (!pool) return GB_ERR_INVALID;
  if (!hidden_dev || !w_dev || hidden_dim <= 0 || hidden_dim % 8 != 0 ||
      (hidden_dtype != GB_F32 && hidden_dtype != GB_BF16))
    return fail(pool, GB_ERR_INVALID, "probe: bad arguments");
  if (((uintptr_t)hidden_dev & 15) || ((uintptr_t)w_dev & 15))
    return fail(pool, GB_ERR_INVALID, "probe: hidden and w must be 16-byte aligned");
  if (pool->next_layer != 0) return fail(pool, GB_ERR_STATE, "probe inside an open step");
  launch_probe(pool, hidden_dev, hidden_dtype, hidden_dim, w_dev, bias, boundary_mask_dev, score_out_dev, nullptr,
               reinterpret_cast<cudaStream_t>(stream));
  return check_launch(pool, "probe");
}

extern "C" gb_status gb_push_scores(gb_pool* pool, const float* scores_dev, const uint8_t* mask_dev,
                                    gb_stream_t stream) {
  if (!pool) return GB_ERR_INVALID;
  if (!scores_dev) return fail(pool, GB_ERR_INVALID, "push_scores: null scores");
  if (pool->next_layer != 0) return fail(pool, GB_ERR_STATE, "push_scores inside an open step");
  launch_probe(pool, nullptr, GB_F32, 8, nullptr, 0.f, mask_dev, nullptr, scores_dev,
               reinterpret_cast<cudaStream_t>(stream));
  return check_launch(pool, "push_scores");
}
