// Two-layer MLP scorer f(h) = sigmoid(w2 . relu(W1 h + b1) + b2) - the light-weight
// 2-layer MLP scorer Gambit is evaluated with (Section 4; Section 3.1: any scorer of the
// last-layer hidden state) - fused with the running-mean update of Algorithm 1.
//
// Layer 1 is the [C x H] . [H x d_h] GEMM Z = H W1^T on the tensor cores:
//   k_mlp_gemm:  grid (C / 128 row tiles) x (d_h / 128 column tiles) x (K splits); each
//                CTA streams its 128 x 64 tiles of H and W1 through a 4-stage TMA ring
//                (128-byte swizzle, K-major) into 128 x 128 x 16 tcgen05.mma (bf16 in,
//                fp32 accumulate in tensor memory) and writes its fp32 partial of Z.
//   k_mlp_score: one CTA per slot: sums the K-split partials in a fixed order, adds b1,
//                applies relu, dots with w2 (deterministic order), adds b2, takes the
//                sigmoid and updates the running mean (subtract, divide, add, each
//                rounded).
// The K split makes about one CTA per SM for any slot count (each split at least four
// 64-wide k-blocks); the partials live in the pool's metadata buffer.  Waits are
// bounded; a timeout records GB_ERR_TIMEOUT.
#include <cuda.h>

#include "internal.cuh"
#include "ptx.cuh"
#include "tc.cuh"

namespace gb {
namespace {

constexpr int kMT = 128, kNT = 128, kKB = 64;  // tile rows (slots), tile columns (d_h), k per stage
constexpr int kMStages = 4;
constexpr int kMStage = 2 * kMT * kKB * 2;      // A and B tiles: 32 KiB
constexpr int kMBar = kMStages * kMStage;
constexpr int kMSmem = kMBar + 128;
constexpr int kMBarFull = 0, kMBarEmpty = 8 * kMStages, kMBarDone = 16 * kMStages;
constexpr int kMWordTmem = kMBarDone + 8;

__device__ __forceinline__ void tma_tile(uint32_t dst, const CUtensorMap* tm, int x, int y, uint32_t bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];" ::"r"(dst),
      "l"(tm), "r"(x), "r"(y), "r"(bar)
      : "memory");
}

__global__ void __launch_bounds__(128, 1)
    k_mlp_gemm(const __grid_constant__ CUtensorMap tmh, const __grid_constant__ CUtensorMap tmw, int rows, int dh,
               int H, float* __restrict__ zp, int* __restrict__ ctl) {
  extern __shared__ __align__(1024) unsigned char sm[];
  if (smem_addr(sm) & 1023) {
    if (threadIdx.x == 0) set_status(ctl, GB_ERR_UNSUPPORTED);
    return;
  }
  const int tid = threadIdx.x, warp = tid >> 5;
  const uint32_t sbase = smem_addr(sm), bar = sbase + kMBar;
  const int mt = blockIdx.x, nt = blockIdx.y, ks = blockIdx.z, splits = gridDim.z;
  const int nkb_all = H / kKB;
  const int kb0 = (int)((long long)ks * nkb_all / splits), kb1 = (int)((long long)(ks + 1) * nkb_all / splits);
  const int nkb = kb1 - kb0;
  if (tid == 0) {
    for (int i = 0; i < kMStages; ++i) {
      mbar_init(bar + kMBarFull + 8 * i, 1);
      mbar_init(bar + kMBarEmpty + 8 * i, 1);
    }
    mbar_init(bar + kMBarDone, 1);
    fence_mbar_init();
  }
  if (warp == 0) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(bar + kMWordTmem),
                 "r"(kNT));
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *reinterpret_cast<volatile uint32_t*>(sm + kMBar + kMWordTmem);
  bool ok = true;
  if (tid == 0) {
    constexpr uint32_t ID = idesc(kMT, kNT, false);
    auto load = [&](int i) {
      const uint32_t st = i % kMStages, full = bar + kMBarFull + 8 * st;
      mbar_arrive_expect_tx(full, kMStage);
      const uint32_t a = sbase + st * kMStage;
      tma_tile(a, &tmh, (kb0 + i) * kKB, mt * kMT, full);
      tma_tile(a + kMT * kKB * 2, &tmw, (kb0 + i) * kKB, nt * kNT, full);
    };
    for (int i = 0; i < nkb && i < kMStages; ++i) load(i);
    for (int i = 0; i < nkb && ok; ++i) {
      const uint32_t st = i % kMStages;
      ok = mbar_wait_bounded(bar + kMBarFull + 8 * st, (i / kMStages) & 1, kWaitLimitNs);
      if (!ok) break;
      tc_fence_after();
      const uint32_t a = sbase + st * kMStage, b = a + kMT * kKB * 2;
#pragma unroll
      for (int kk = 0; kk < kKB / 16; ++kk)
        mma(tmem, sdesc(a + kk * 32, 16, 1024), sdesc(b + kk * 32, 16, 1024), ID, (i > 0 || kk > 0) ? 1u : 0u);
      mma_commit(bar + kMBarEmpty + 8 * st);
      if (i + kMStages < nkb) {  // refill this stage once its MMAs have read it
        ok = mbar_wait_bounded(bar + kMBarEmpty + 8 * st, (i / kMStages) & 1, kWaitLimitNs);
        if (ok) load(i + kMStages);
      }
    }
    if (ok) mma_commit(bar + kMBarDone);
    if (!ok) set_status(ctl, GB_ERR_TIMEOUT);
  }
  __syncthreads();
  ok = __syncthreads_and(tid == 0 ? ok : 1);
  // Thread r writes row r of the partial tile (fp32), columns inside d_h only.
  const int r = tid, row = mt * kMT + r;
  if (ok && nkb > 0 && mbar_wait_bounded(bar + kMBarDone, 0, kWaitLimitNs)) {
    tc_fence_after();
    float* dst = zp + ((size_t)ks * rows + row) * dh + (size_t)nt * kNT;
#pragma unroll 1
    for (int c0 = 0; c0 < kNT; c0 += 32) {
      float z[32];
      tmem_ld32(tmem + ((uint32_t)(warp * 32) << 16) + c0, z);
      if (row < rows) {
#pragma unroll
        for (int i = 0; i < 32; ++i)
          if (nt * kNT + c0 + i < dh) dst[c0 + i] = z[i];
      }
    }
  } else if (nkb == 0 && row < rows) {
    float* dst = zp + ((size_t)ks * rows + row) * dh + (size_t)nt * kNT;
    for (int c = 0; c < kNT && nt * kNT + c < dh; ++c) dst[c] = 0.f;
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kNT));
}

// One CTA per slot: thread t sums the K-split partials of columns t, t + blockDim, ...
// (consecutive threads read consecutive columns), applies b1 and relu, weights by w2;
// the block reduces in a fixed order.
constexpr int kScoreThreads = 256;

__global__ void __launch_bounds__(kScoreThreads) k_mlp_score(PoolView v, const float* __restrict__ zp, int splits,
                                                             int dh, const float* __restrict__ b1,
                                                             const float* __restrict__ w2, float b2,
                                                             const uint8_t* __restrict__ mask,
                                                             float* __restrict__ score_out) {
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

typedef CUresult (*EncodeFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*, const cuuint64_t*,
                             const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                             CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

// 2D bf16 tensor map over a [rows][cols] row-major matrix: box 64 columns x 128 rows, 128-byte swizzle.
bool encode_rows(CUtensorMap* m, const void* base, int rows, int cols) {
  static EncodeFn encode = nullptr;
  if (!encode) {
    cudaDriverEntryPointQueryResult qr;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", reinterpret_cast<void**>(&encode), 12000,
                                         cudaEnableDefault, &qr) != cudaSuccess ||
        qr != cudaDriverEntryPointSuccess || !encode)
      return false;
  }
  cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
  cuuint64_t strides[1] = {(cuuint64_t)cols * 2};
  cuuint32_t box[2] = {kKB, kMT};
  cuuint32_t es[2] = {1, 1};
  return encode(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, es,
                CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace

cudaError_t launch_mlp(gb_pool* pool, const void* hidden, int H, const void* w1, const float* b1, const float* w2,
                       float b2, int dh, const uint8_t* mask, float* score_out, cudaStream_t s) {
  static bool configured = false;
  if (!configured) {
    cudaError_t e = cudaFuncSetAttribute(k_mlp_gemm, cudaFuncAttributeMaxDynamicSharedMemorySize, kMSmem);
    if (e != cudaSuccess) return e;
    configured = true;
  }
  const PoolView& v = pool->view;
  CUtensorMap th, tw;
  if (!encode_rows(&th, hidden, v.max_beams, H) || !encode_rows(&tw, w1, dh, H)) return cudaErrorInvalidValue;
  const int mtiles = (v.max_beams + kMT - 1) / kMT, ntiles = (dh + kNT - 1) / kNT;
  // About one CTA per SM, each split at least 4 k-blocks deep.
  const int nkb = H / kKB;
  int splits = pool->num_sms / (mtiles * ntiles);
  splits = splits > nkb / 4 ? nkb / 4 : splits;
  splits = splits < 1 ? 1 : splits;
  while (splits > 1 && (size_t)splits * v.max_beams * dh > (size_t)kMlpScratchFloats) --splits;
  if ((size_t)splits * v.max_beams * dh > (size_t)kMlpScratchFloats) return cudaErrorInvalidValue;
  prof_begin(pool, GB_PROF_PROBE, s);
  k_mlp_gemm<<<dim3(mtiles, ntiles, splits), 128, kMSmem, s>>>(th, tw, v.max_beams, dh, H, v.mlp_scratch, v.ctl);
  k_mlp_score<<<v.max_beams, kScoreThreads, 0, s>>>(v, v.mlp_scratch, splits, dh, b1, w2, b2, mask, score_out);
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
