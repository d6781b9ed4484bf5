// Scorer probe f(h) = sigmoid(w.h + b) fused with the running-mean update of
// Algorithm 1 ("s_bar <- s_bar + (f(h_n) - s_bar)/n").  One warp per slot:
// 16-byte loads of the hidden row, fp32 accumulation, shuffle reduction.
// The mean update rounds subtract, divide and add separately, in that order.
#include "internal.cuh"

namespace gb {

template <int HT>
__device__ __forceinline__ float dot_row(const void* hrow, const float* __restrict__ w, int H, int lane) {
  float acc = 0.f;
  if constexpr (HT == GB_BF16) {
    const uint4* h4 = static_cast<const uint4*>(hrow);
    for (int e = lane; e < H / 8; e += 32) {
      const uint4 u = h4[e];
      const float4 wa = reinterpret_cast<const float4*>(w)[2 * e];
      const float4 wb = reinterpret_cast<const float4*>(w)[2 * e + 1];
      acc = fmaf(__uint_as_float(u.x << 16), wa.x, acc);
      acc = fmaf(__uint_as_float(u.x & 0xffff0000u), wa.y, acc);
      acc = fmaf(__uint_as_float(u.y << 16), wa.z, acc);
      acc = fmaf(__uint_as_float(u.y & 0xffff0000u), wa.w, acc);
      acc = fmaf(__uint_as_float(u.z << 16), wb.x, acc);
      acc = fmaf(__uint_as_float(u.z & 0xffff0000u), wb.y, acc);
      acc = fmaf(__uint_as_float(u.w << 16), wb.z, acc);
      acc = fmaf(__uint_as_float(u.w & 0xffff0000u), wb.w, acc);
    }
  } else {
    const float4* h4 = static_cast<const float4*>(hrow);
    for (int e = lane; e < H / 4; e += 32) {
      const float4 u = h4[e];
      const float4 wa = reinterpret_cast<const float4*>(w)[e];
      acc = fmaf(u.x, wa.x, acc);
      acc = fmaf(u.y, wa.y, acc);
      acc = fmaf(u.z, wa.z, acc);
      acc = fmaf(u.w, wa.w, acc);
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
  return acc;
}

template <int HT>
__global__ void k_probe(PoolView v, const void* __restrict__ hidden, int H, const float* __restrict__ w,
                        float bias, const uint8_t* __restrict__ mask, float* __restrict__ score_out,
                        const float* __restrict__ scores_in) {
  pdl_wait();
  pdl_launch_dependents();
  const int lane = threadIdx.x & 31;
  const int warps = blockDim.x >> 5;
  for (int b = blockIdx.x * warps + (threadIdx.x >> 5); b < v.max_beams; b += gridDim.x * warps) {
    if (!v.active[b]) {
      if (score_out && lane == 0) score_out[b] = 0.f;
      continue;
    }
    float x;
    if (scores_in) {
      x = scores_in[b];
    } else {
      const size_t es = HT == GB_BF16 ? 2 : 4;
      const float z = dot_row<HT>(static_cast<const char*>(hidden) + (size_t)b * H * es, w, H, lane) + bias;
      x = 1.0f / (1.0f + expf(-z));
      if (score_out && lane == 0) score_out[b] = x;
    }
    if (lane == 0 && (mask == nullptr || mask[b] != 0)) {
      const int n = v.nsteps[b] + 1;
      const float m = v.mean[b];
      const float d = __fsub_rn(x, m);
      const float q = __fdiv_rn(d, (float)n);
      v.mean[b] = __fadd_rn(m, q);
      v.nsteps[b] = n;
    }
  }
}

cudaError_t launch_probe(gb_pool* pool, const void* hidden, int hidden_dtype, int H, const float* w, float bias,
                         const uint8_t* mask, float* score_out, const float* scores_in, cudaStream_t s) {
  const int warps_per_block = 8;
  const int grid = (pool->view.max_beams + warps_per_block - 1) / warps_per_block;
  pool->launches += 1;
  if (scores_in == nullptr) prof_begin(pool, GB_PROF_PROBE, s);
  const cudaError_t e =
      hidden_dtype == GB_BF16
          ? launch_pdl(k_probe<GB_BF16>, grid, warps_per_block * 32, 0, s, pool->view, hidden, H, w, bias, mask,
                       score_out, scores_in)
          : launch_pdl(k_probe<GB_F32>, grid, warps_per_block * 32, 0, s, pool->view, hidden, H, w, bias, mask,
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
