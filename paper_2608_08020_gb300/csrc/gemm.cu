// Split-K bf16 GEMM on tcgen05 for the scorers: P[s][m][n] = sum over the s-th k-range of
// A[m][k] * B[n][k] (A [M][K] and B [N][K] bf16 row-major, fp32 partials).
// Grid (M / 128) x (N / 128) x splits; one thread streams 128 x 64 tiles of A and B
// through a 4-stage TMA ring (2D tensor maps, 128-byte swizzle, K-major) into
// 128 x 128 x 16 tcgen05.mma accumulating in tensor memory; the CTA writes its partial
// tile (rows < M, columns < N).  Out-of-range rows and columns load as zeros.  Waits are
// bounded; a timeout records GB_ERR_TIMEOUT in the caller's status word.
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
    k_gemm_partials(const __grid_constant__ CUtensorMap tmh, const __grid_constant__ CUtensorMap tmw, int rows, int dh,
               int H, float* __restrict__ zp, int* __restrict__ ctl) {
  pdl_wait();
  pdl_launch_dependents();
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
  // The partial tile goes out through shared memory (the ring is idle once the MMAs are
  // done): thread r reads row r's 32 columns of a chunk from TMEM into a padded tile, then
  // each warp stores whole rows, lanes over consecutive columns (rows < M, columns < N).
  const int r = tid, lane = tid & 31;
  float* stile = reinterpret_cast<float*>(sm);  // [128][33]
  float* base = zp + (size_t)ks * rows * dh;
  const bool done = ok && nkb > 0 && mbar_wait_bounded(bar + kMBarDone, 0, kWaitLimitNs);
  const bool have = __syncthreads_and(done);  // uniform: tcgen05.ld is warp-collective
  if (ok && nkb > 0 && !have && tid == 0) set_status(ctl, GB_ERR_TIMEOUT);
  if (have) tc_fence_after();
#pragma unroll 1
  for (int c0 = 0; c0 < kNT; c0 += 32) {
    if (nt * kNT + c0 >= dh) break;
    if (have) {
      float z[32];
      tmem_ld32(tmem + ((uint32_t)(warp * 32) << 16) + c0, z);
#pragma unroll
      for (int i = 0; i < 32; ++i) stile[r * 33 + i] = z[i];
    }
    __syncthreads();
    const int col = nt * kNT + c0 + lane;
    for (int rr = warp; rr < kMT; rr += 4) {
      const int row = mt * kMT + rr;
      if (row < rows && col < dh) base[(size_t)row * dh + col] = have ? stile[rr * 33 + lane] : 0.f;
    }
    __syncthreads();
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kNT));
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

int gemm_splits(int M, int N, int K, int num_sms, size_t max_floats) {
  const int mtiles = (M + kMT - 1) / kMT, ntiles = (N + kNT - 1) / kNT;
  const int nkb = K / kKB;
  // About one CTA per SM, each split at least 4 k-blocks deep, partials within max_floats.
  int splits = num_sms / (mtiles * ntiles);
  splits = splits > nkb / 4 ? nkb / 4 : splits;
  splits = splits < 1 ? 1 : splits;
  while (splits > 1 && (size_t)splits * M * N > max_floats) --splits;
  return (size_t)splits * M * N > max_floats ? 0 : splits;
}

cudaError_t gemm_partials(const void* A, int M, const void* B, int N, int K, int splits, float* P, int* ctl,
                          cudaStream_t s) {
  {
    const cudaError_t e = set_max_dynamic_smem(reinterpret_cast<const void*>(k_gemm_partials), kMSmem);
    if (e != cudaSuccess) return e;
  }
  if (K % kKB != 0 || splits < 1) return cudaErrorInvalidValue;
  CUtensorMap ta, tb;
  if (!encode_rows(&ta, A, M, K) || !encode_rows(&tb, B, N, K)) return cudaErrorInvalidValue;
  const int mtiles = (M + kMT - 1) / kMT, ntiles = (N + kNT - 1) / kNT;
  return launch_pdl(k_gemm_partials, dim3(mtiles, ntiles, splits), 128, kMSmem, s, ta, tb, M, N, K, P, ctl);
}

}  // namespace gb
