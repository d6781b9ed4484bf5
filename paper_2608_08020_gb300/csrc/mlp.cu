// Two-layer MLP scorer f(h) = sigmoid(w2 . relu(W1 h + b1) + b2) - the light-weight
// 2-layer MLP scorer Gambit is evaluated with (Section 4; Section 3.1: any scorer of the
// last-layer hidden state) - fused with the running-mean update of Algorithm 1.
//
// Layer 1 is the [C x H] . [H x d_h] GEMM Z = H W1^T on the tensor cores (gemm.cu: a
// split-K tcgen05 GEMM writing fp32 partials of Z), then
//   k_mlp_score: one CTA per slot: sums the K-split partials in a fixed order, adds b1,
//                applies relu, dots with w2 (deterministic order), adds b2, takes the
//                sigmoid and updates the running mean (subtract, divide, add, each
//                rounded).
// The K split makes about one CTA per SM for any slot count (each split at least four
// 64-wide k-blocks); the partials live in the pool's metadata buffer.  Waits are
// bounded; a timeout records GB_ERR_TIMEOUT.
#include "internal.cuh"

namespace gb {
namespace {

// One CTA per slot: thread t sums the K-split partials of columns t, t + blockDim, ...
// (consecutive threads read consecutive columns), applies b1 and relu, weights by w2;
// the block reduces in a fixed order.
constexpr int kScoreThreads = 256;

__global__ void __launch_bounds__(kScoreThreads) k_mlp_score(PoolView v, const float* __restrict__ zp, int splits,
                                                             int dh, const float* __restrict__ b1,
                                                             const float* __restrict__ w2, float b2,
                                                             const uint8_t* __restrict__ mask,
                                                             float* __restrict__ score_out) {
  pdl_wait();
  pdl_launch_dependents();
  __shared__ float red[kScoreThreads / 32];
  const int b = blockIdx.x, tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  if (!v.active[b]) {
    if (score_out && tid == 0) score_out[b] = 0.f;
    return;
  }
  float acc = 0.f;
  for (int n = tid; n < dh; n += kScoreThreads) {
    float z = b1[n];
    for (int k = 0; k < splits; ++k) z += zp[((size_t)k * v.max_beams + b) * dh + n];
    acc = fmaf(fmaxf(z, 0.f), w2[n], acc);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
  if (lane == 0) red[warp] = acc;
  __syncthreads();
  if (tid == 0) {
    float y = 0.f;
    for (int w = 0; w < kScoreThreads / 32; ++w) y += red[w];
    const float x = 1.0f / (1.0f + expf(-(y + b2)));
    if (score_out) score_out[b] = x;
    if (mask == nullptr || mask[b] != 0) {
      const int n = v.nsteps[b] + 1;
      const float m = v.mean[b];
      v.mean[b] = __fadd_rn(m, __fdiv_rn(__fsub_rn(x, m), (float)n));
      v.nsteps[b] = n;
    }
  }
}

}  // namespace

cudaError_t launch_mlp(gb_pool* pool, const void* hidden, int H, const void* w1, const float* b1, const float* w2,
                       float b2, int dh, const uint8_t* mask, float* score_out, cudaStream_t s) {
  const PoolView& v = pool->view;
  const int splits = gemm_splits(v.max_beams, dh, H, pool->num_sms, kMlpScratchFloats);
  if (splits == 0) return cudaErrorInvalidValue;
  prof_begin(pool, GB_PROF_PROBE, s);
  cudaError_t e = gemm_partials(hidden, v.max_beams, w1, dh, H, splits, v.mlp_scratch, v.ctl, s);
  if (e != cudaSuccess) return e;
  e = launch_pdl(k_mlp_score, v.max_beams, kScoreThreads, 0, s, v, static_cast<const float*>(v.mlp_scratch), splits,
                 dh, b1, w2, b2, mask, score_out);
  if (e != cudaSuccess) return e;
  prof_end(pool, GB_PROF_PROBE, s);
  pool->launches += 2;
  return cudaGetLastError();
}

}  // namespace gb

using namespace gb;

extern "C" gb_status gb_score_mlp(gb_pool* pool, const void* hidden_dev, int hidden_dim, const void* w1_dev,
                                  const float* b1_dev, const float* w2_dev, float b2, int d_h,
                                  const uint8_t* boundary_mask_dev, float* score_out_dev, gb_stream_t stream) {
  if (!pool) return GB_ERR_INVALID;
  if (!hidden_dev || !w1_dev || !b1_dev || !w2_dev || hidden_dim <= 0 || hidden_dim % 64 != 0 || d_h <= 0)
    return fail(pool, GB_ERR_INVALID, "score_mlp: bad arguments");
  if (((uintptr_t)hidden_dev & 15) || ((uintptr_t)w1_dev & 15))
    return fail(pool, GB_ERR_INVALID, "score_mlp: hidden and w1 must be 16-byte aligned");
  if ((size_t)pool->view.max_beams * d_h > (size_t)kMlpScratchFloats)
    return fail(pool, GB_ERR_TOO_LARGE, "score_mlp: max_beams x d_h exceeds the partial-sum buffer");
  if (pool->next_layer != 0) return fail(pool, GB_ERR_STATE, "score_mlp inside an open step");
  if (launch_mlp(pool, hidden_dev, hidden_dim, w1_dev, b1_dev, w2_dev, b2, d_h, boundary_mask_dev, score_out_dev,
                 reinterpret_cast<cudaStream_t>(stream)) != cudaSuccess)
    return check_launch(pool, "score_mlp");
  return check_launch(pool, "score_mlp");
}
