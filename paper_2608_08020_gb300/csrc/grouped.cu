// Grouped shared-prefix decode attention on tcgen05 tensor cores.
//
// For a segment of pages shared by g beams, the g x G query rows of one KV head
// (G = Hq / Hkv) are stacked into one 128-row tile, so the segment's K and V are
// read once for all of them and Q.K^T and P.V become dense contractions:
//   S[128 x 64]  = Q[128 x 128] . K_tile^T      (tcgen05.mma kind::f16, fp32 in TMEM)
//   O[128 x 128] += P[128 x 64] . V_tile         (P in bf16 from the softmax)
// over 64-token tiles of the segment.  Each unit of work is (segment, KV head,
// 128-row query tile); a persistent grid of one CTA per SM walks the flat unit list.
// Results are unnormalised partials (m, l, o) per (beam, depth, head) merged by the
// combine kernel with the beam's per-beam remainder.
//
// Shared memory (1024-byte aligned, 128-byte swizzle everywhere):
//   Q   two [128 rows][64 dims] blocks (K-major A operand)             32 KiB
//   K,V per stage: two [64 tokens][64 dims] blocks each               32 KiB x 2 stages
//   P   one [128 rows][64 tokens] block (K-major A operand)           16 KiB
// K/V chunks of 16 tokens arrive by 2D TMA loads (box 64 dims x 16 rows) from a
// tensor map over the whole pool; chunks past the segment end load out of bounds
// and are zero-filled.  V is the B operand in MN-major form (dims contiguous).
//
// Softmax: thread r owns row r (TMEM lane r).  The running maximum is only raised
// when a tile's maximum exceeds it by more than 8 (base 2); smaller increases are
// absorbed in p <= 2^8, so O in TMEM is rescaled rarely.  Every mbarrier wait is
// bounded; on timeout the CTA records GB_ERR_TIMEOUT, drains its own copies and
// MMAs (bounded), frees its tensor memory and leaves.
#include <cuda.h>

#include "internal.cuh"
#include "ptx.cuh"

namespace gb {
namespace {

constexpr int kRows = 128;     // query rows per tile (MMA M)
constexpr int kTok = 64;       // tokens per K/V tile (MMA N of Q.K^T, K of P.V)
constexpr int kStages = 4;
constexpr int kThreads = 128;
constexpr uint32_t kTmemCols = 256;  // S: columns [0, 64), O: [128, 256)

constexpr int kQ = 0;
constexpr int kKV = 32768;
constexpr int kStage = 32768;        // K 16 KiB + V 16 KiB
constexpr int kP = kKV + kStages * kStage;
constexpr int kSmem = kP + 16384;
constexpr int kSmemAlloc = kSmem + 1024;

__device__ __forceinline__ uint32_t swz(int r, int col) {  // byte offset of (row, col) in a [rows][64] bf16 SW128 block
  return (uint32_t)((r >> 3) * 1024 + (r & 7) * 128 + ((((col >> 3) ^ (r & 7))) << 4) + (col & 7) * 2);
}

__device__ __forceinline__ uint64_t sdesc(uint32_t addr, uint32_t lbo, uint32_t sbo) {
  uint64_t d = (uint64_t)((addr >> 4) & 0x3FFF);
  d |= (uint64_t)((lbo >> 4) & 0x3FFF) << 16;
  d |= (uint64_t)((sbo >> 4) & 0x3FFF) << 32;
  d |= (uint64_t)1 << 46;  // descriptor version for tcgen05
  d |= (uint64_t)2 << 61;  // 128-byte swizzle
  return d;
}

// kind::f16 instruction descriptor: bf16 A and B, fp32 accumulate, M = 128.
__host__ __device__ constexpr uint32_t idesc(int n, bool b_mn_major) {
  return (1u << 4) | (1u << 7) | (1u << 10) | ((b_mn_major ? 1u : 0u) << 16) | ((uint32_t)(n >> 3) << 17) |
         ((uint32_t)(kRows >> 4) << 24);
}

__device__ __forceinline__ void mma(uint32_t tmem_d, uint64_t a, uint64_t b, uint32_t id, uint32_t acc) {
  asm volatile(
      "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(tmem_d),
      "l"(a), "l"(b), "r"(id), "r"(acc));
}

__device__ __forceinline__ void mma_commit(uint32_t bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar) : "memory");
}

__device__ __forceinline__ void tma_2d(uint32_t dst, const CUtensorMap* tm, int x, int y, uint32_t bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];" ::"r"(dst),
      "l"(tm), "r"(x), "r"(y), "r"(bar)
      : "memory");
}

__device__ __forceinline__ void tmem_ld32(uint32_t taddr, float* f) {
  uint32_t r[32];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
      "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]), "=r"(r[8]),
        "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]),
        "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]),
        "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr));
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
  for (int i = 0; i < 32; ++i) f[i] = __uint_as_float(r[i]);
}

__device__ __forceinline__ void tmem_st32(uint32_t taddr, const float* f) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,"
      "%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32};" ::"r"(taddr),
      "r"(__float_as_uint(f[0])), "r"(__float_as_uint(f[1])), "r"(__float_as_uint(f[2])), "r"(__float_as_uint(f[3])),
      "r"(__float_as_uint(f[4])), "r"(__float_as_uint(f[5])), "r"(__float_as_uint(f[6])), "r"(__float_as_uint(f[7])),
      "r"(__float_as_uint(f[8])), "r"(__float_as_uint(f[9])), "r"(__float_as_uint(f[10])), "r"(__float_as_uint(f[11])),
      "r"(__float_as_uint(f[12])), "r"(__float_as_uint(f[13])), "r"(__float_as_uint(f[14])), "r"(__float_as_uint(f[15])),
      "r"(__float_as_uint(f[16])), "r"(__float_as_uint(f[17])), "r"(__float_as_uint(f[18])), "r"(__float_as_uint(f[19])),
      "r"(__float_as_uint(f[20])), "r"(__float_as_uint(f[21])), "r"(__float_as_uint(f[22])), "r"(__float_as_uint(f[23])),
      "r"(__float_as_uint(f[24])), "r"(__float_as_uint(f[25])), "r"(__float_as_uint(f[26])), "r"(__float_as_uint(f[27])),
      "r"(__float_as_uint(f[28])), "r"(__float_as_uint(f[29])), "r"(__float_as_uint(f[30])), "r"(__float_as_uint(f[31]))
      : "memory");
  asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
}

__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }

template <int G>
__global__ void __launch_bounds__(kThreads, 1)
    k_grouped(PoolView v, const __grid_constant__ CUtensorMap tm, int layer, const __nv_bfloat16* __restrict__ q,
              float qscale, long long total_rows) {
  extern __shared__ __align__(1024) unsigned char smem_raw[];
  unsigned char* sm = reinterpret_cast<unsigned char*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  __shared__ __align__(8) uint64_t bar_full[kStages];
  __shared__ __align__(8) uint64_t bar_s, bar_pv;
  __shared__ uint32_t tmem_slot;
  __shared__ int s_abort;

  if (v.ctl[kCtlStepOk] == 0) return;
  const int ntiles_q = v.ctl[kCtlSegTiles];
  const long long units = (long long)ntiles_q * v.Hkv;
  if (blockIdx.x >= units) return;

  const int tid = threadIdx.x, warp = tid >> 5;
  const uint32_t sbase = smem_addr(sm);
  const uint32_t bfull0 = smem_addr(&bar_full[0]);
  const uint32_t bs = smem_addr(&bar_s), bpv = smem_addr(&bar_pv);
  if (tid == 0) {
    for (int i = 0; i < kStages; ++i) mbar_init(bfull0 + 8 * i, 1);
    mbar_init(bs, 1);
    mbar_init(bpv, 1);
    fence_mbar_init();
    s_abort = 0;
  }
  if (warp == 0) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_addr(&tmem_slot)),
                 "r"(kTmemCols));
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tmem_slot;
  const uint32_t tS = tmem, tO = tmem + 128;
  const uint32_t lane_base = (uint32_t)(warp * 32) << 16;

  constexpr uint32_t ID_S = idesc(kTok, false);
  constexpr uint32_t ID_PV = idesc(128, true);
  const long long rows_per_kvhead = (long long)v.P;  // tensor-map rows of one (layer, page, kv, head) slab

  // Per-CTA pipeline counters (continue across units).
  uint32_t loads_issued = 0, loads_used = 0, s_done = 0, pv_done = 0;
  bool timed_out = false;

  auto issue_tile = [&](int seg_i0, int tok_base, int rep, int h, int Ts, int j, uint32_t stage) {
    // Tokens [64j, 64j+64) of the segment: four 16-token chunks, K and V, two 64-dim halves.
    const uint32_t bar = bfull0 + 8 * stage;
    mbar_arrive_expect_tx(bar, kStage);
    const uint32_t dst0 = sbase + kKV + stage * kStage;
#pragma unroll
    for (int c = 0; c < 4; ++c) {
      const int tk = tok_base + j * kTok + c * 16;  // token within the segment
      long long yk = total_rows, yv = total_rows;  // out of bounds: zero fill
      if (j * kTok + c * 16 < Ts) {
        int page = v.tables[(size_t)rep * v.max_pages + seg_i0 + tk / v.P];
        if (page < 0 || page >= v.num_pages) {
          set_status(v.ctl, GB_ERR_INVALID);
          page = 0;
        }
        const long long slab = (((long long)layer * v.num_pages + page) * 2) * v.Hkv + h;
        yk = slab * rows_per_kvhead + tk % v.P;
        yv = (slab + v.Hkv) * rows_per_kvhead + tk % v.P;
      }
#pragma unroll
      for (int half = 0; half < 2; ++half) {
        tma_2d(dst0 + half * 8192 + c * 2048, &tm, half * 64, (int)yk, bar);
        tma_2d(dst0 + 16384 + half * 8192 + c * 2048, &tm, half * 64, (int)yv, bar);
      }
    }
  };

  for (long long u = blockIdx.x; u < units && !timed_out; u += gridDim.x) {
    const int tq = (int)(u / v.Hkv), h = (int)(u % v.Hkv);
    const int s = v.seg_tile_seg[tq], t = v.seg_tile_t[tq], sp = v.seg_tile_split[tq];
    const int split = v.ctl[kCtlSegSplit];
    const int tok_base = sp * split;
    const int seg_i0 = v.seg_i0[s], rep = v.seg_rep[s], g = v.seg_g[s], moff = v.seg_mem_off[s];
    const int Ts = min(v.seg_len[s] * v.P - tok_base, split);  // tokens of this split
    const int ntok = (Ts + kTok - 1) / kTok;
    constexpr int members_per_tile = kRows / G;

    // Q tile: row r = (member, query head of this KV head), zero rows past the members.
    {
      const int r = tid;
      const int m = t * members_per_tile + r / G, gg = r % G;
      const bool valid = m < g;
      const int bk = valid ? v.seg_members[moff + m] : 0;
      const int b = bk / kMaxSegDepth;
      const uint4* qrow = reinterpret_cast<const uint4*>(q + ((size_t)b * v.Hq + (size_t)h * G + gg) * 128);
#pragma unroll
      for (int c = 0; c < 16; ++c) {
        const uint4 x = valid ? qrow[c] : make_uint4(0, 0, 0, 0);
        *reinterpret_cast<uint4*>(sm + kQ + (c >> 3) * 16384 + swz(r, (c & 7) * 8)) = x;
      }
    }
    fence_proxy_async_smem();
    tc_fence_before();
    __syncthreads();
    tc_fence_after();

    if (tid == 0) {
      for (int j = 0; j < kStages && j < ntok; ++j) issue_tile(seg_i0, tok_base, rep, h, Ts, j, (loads_issued + j) % kStages);
    }
    uint32_t issued_here = ntok < kStages ? ntok : kStages;

    // S(0)
    auto issue_s = [&](uint32_t stage) {
      const uint32_t kb = sbase + kKV + stage * kStage;
#pragma unroll
      for (int kk = 0; kk < 8; ++kk) {
        const uint64_t a = sdesc(sbase + kQ + (kk >> 2) * 16384 + (kk & 3) * 32, 16, 1024);
        const uint64_t b = sdesc(kb + (kk >> 2) * 8192 + (kk & 3) * 32, 16, 1024);
        mma(tS, a, b, ID_S, kk > 0);
      }
      mma_commit(bs);
    };
    if (tid == 0) {
      const uint32_t st = loads_issued % kStages;
      if (!mbar_wait_bounded(bfull0 + 8 * st, (loads_issued / kStages) & 1, kWaitLimitNs)) {
        s_abort = 1;
      } else {
        tc_fence_after();
        issue_s(st);
      }
    }

    float m_ref = -INFINITY, l = 0.f;
    for (int j = 0; j < ntok; ++j) {
      const uint32_t gj = loads_used + j;           // global tile counter of this CTA
      const uint32_t stage = gj % kStages;
      // Wait for S(j).
      if (!mbar_wait_bounded(bs, s_done & 1, kWaitLimitNs)) { timed_out = true; }
      if (__syncthreads_or(timed_out || s_abort)) { timed_out = true; break; }
      ++s_done;
      tc_fence_after();
      float sv[kTok];
      tmem_ld32(tS + lane_base + 0, sv);
      tmem_ld32(tS + lane_base + 32, sv + 32);
      float mt = -INFINITY;
#pragma unroll
      for (int c = 0; c < kTok; ++c) {
        const bool ok = j * kTok + c < Ts;
        sv[c] = ok ? sv[c] * qscale : -INFINITY;
        mt = fmaxf(mt, sv[c]);
      }
      // P.V of the previous tile must be done before P and O are touched and its stage refilled.
      if (j > 0) {
        if (!mbar_wait_bounded(bpv, pv_done & 1, kWaitLimitNs)) timed_out = true;
        if (__syncthreads_or(timed_out)) { timed_out = true; break; }
        ++pv_done;
        tc_fence_after();
        if (tid == 0 && j - 1 + kStages < ntok) {
          issue_tile(seg_i0, tok_base, rep, h, Ts, j - 1 + kStages, (gj - 1) % kStages);
          ++issued_here;
        }
      }
      const bool raise = mt > m_ref + 8.f;
      if (j > 0 && __any_sync(0xffffffffu, raise)) {
        const float alpha = raise ? exp2f(m_ref - mt) : 1.f;
#pragma unroll 1
        for (int c0 = 0; c0 < 128; c0 += 32) {
          float o[32];
          tmem_ld32(tO + lane_base + c0, o);
#pragma unroll
          for (int i = 0; i < 32; ++i) o[i] *= alpha;
          tmem_st32(tO + lane_base + c0, o);
        }
        if (raise) l *= alpha;
      }
      if (raise) m_ref = mt;
      // p = 2^(s - m_ref) in bf16 into the P tile (row = tid), l accumulates the same rounded values.
#pragma unroll
      for (int c = 0; c < kTok; c += 8) {
        __nv_bfloat162 pr[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          pr[i] = __floats2bfloat162_rn(exp2f(sv[c + 2 * i] - m_ref), exp2f(sv[c + 2 * i + 1] - m_ref));
          const float2 back = __bfloat1622float2(pr[i]);
          l += back.x + back.y;
        }
        *reinterpret_cast<uint4*>(sm + kP + swz(tid, c)) = *reinterpret_cast<const uint4*>(pr);
      }
      fence_proxy_async_smem();
      tc_fence_before();
      __syncthreads();
      if (tid == 0) {
        tc_fence_after();
        const uint32_t vb = sbase + kKV + stage * kStage + 16384;
#pragma unroll
        for (int kk = 0; kk < kTok / 16; ++kk) {
          const uint64_t a = sdesc(sbase + kP + kk * 32, 16, 1024);
          const uint64_t b = sdesc(vb + kk * 2048, 8192, 1024);
          mma(tO, a, b, ID_PV, (j > 0 || kk > 0) ? 1u : 0u);
        }
        mma_commit(bpv);
        if (j + 1 < ntok) {
          const uint32_t st = (gj + 1) % kStages;
          if (!mbar_wait_bounded(bfull0 + 8 * st, ((gj + 1) / kStages) & 1, kWaitLimitNs)) {
            s_abort = 1;
          } else {
            tc_fence_after();
            issue_s(st);
          }
        }
      }
    }
    if (timed_out) break;
    // Final P.V, then write this tile's rows.
    if (!mbar_wait_bounded(bpv, pv_done & 1, kWaitLimitNs)) timed_out = true;
    if (__syncthreads_or(timed_out)) { timed_out = true; break; }
    ++pv_done;
    tc_fence_after();
    loads_used += ntok;
    loads_issued += ntok;
    {
      const int r = tid;
      const int m = t * members_per_tile + r / G, gg = r % G;
      const int bk = m < g ? v.seg_members[moff + m] : 0;
      const int b = bk / kMaxSegDepth;
      const int r_idx = v.seg_rec_off[bk] + sp;
      const bool has = m < g && r_idx < kMaxSegRecords;
      float* rec = v.grec + (((size_t)b * kMaxSegRecords + r_idx) * v.Hkv + h) * v.record_floats;
#pragma unroll 1
      for (int c0 = 0; c0 < 128; c0 += 32) {  // warp-collective loads: every lane takes part
        float o[32];
        tmem_ld32(tO + lane_base + c0, o);
        if (has) {
#pragma unroll
          for (int i = 0; i < 32; i += 4)
            *reinterpret_cast<float4*>(rec + gg * 128 + c0 + i) = make_float4(o[i], o[i + 1], o[i + 2], o[i + 3]);
        }
      }
      if (has) {
        rec[G * 128 + gg] = m_ref;
        rec[G * 128 + G + gg] = l;
      }
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
  }

  if (timed_out) {
    if (tid == 0) {
      set_status(v.ctl, GB_ERR_TIMEOUT);
      // Give this CTA's outstanding copies and MMAs a bounded chance to finish before leaving.
      for (int i = 0; i < kStages; ++i) mbar_wait_bounded(bfull0 + 8 * i, 0, kWaitLimitNs / 8);
      mbar_wait_bounded(bs, s_done & 1, kWaitLimitNs / 8);
      mbar_wait_bounded(bpv, pv_done & 1, kWaitLimitNs / 8);
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kTmemCols));
}

}  // namespace

// 2D tensor map over the whole pool: rows of D = 128 bf16 (256 bytes), box 64 x 16, 128-byte swizzle.
bool make_kv_tensor_map(gb_pool* pool) {
  typedef CUresult (*EncodeFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                               const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                               CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);
  static EncodeFn encode = nullptr;
  if (!encode) {
    cudaDriverEntryPointQueryResult qr;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", reinterpret_cast<void**>(&encode), 12000,
                                         cudaEnableDefault, &qr) != cudaSuccess ||
        qr != cudaDriverEntryPointSuccess || !encode)
      return false;
  }
  const PoolView& v = pool->view;
  const unsigned long long rows = (unsigned long long)v.layers * v.num_pages * 2 * v.Hkv * v.P;
  if (rows >= (1ull << 31)) return false;
  cuuint64_t dims[2] = {128, rows};
  cuuint64_t strides[1] = {256};
  cuuint32_t box[2] = {64, 16};
  cuuint32_t es[2] = {1, 1};
  CUtensorMap* m = reinterpret_cast<CUtensorMap*>(pool->tmap);
  const CUresult r = encode(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, v.kv, dims, strides, box, es,
                            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  pool->have_tmap = r == CUDA_SUCCESS;
  return pool->have_tmap;
}

template <int G>
static cudaError_t launch_grouped_t(gb_pool* pool, int layer, const void* q, float scale, cudaStream_t s) {
  static bool configured = false;
  if (!configured) {
    cudaError_t e = cudaFuncSetAttribute(k_grouped<G>, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemAlloc);
    if (e != cudaSuccess) return e;
    configured = true;
  }
  const PoolView& v = pool->view;
  const long long rows = (long long)v.layers * v.num_pages * 2 * v.Hkv * v.P;
  const float qscale = scale * 1.4426950408889634f;
  prof_begin(pool, GB_PROF_GROUPED, s);
  k_grouped<G><<<pool->num_sms, kThreads, kSmemAlloc, s>>>(
      v, *reinterpret_cast<const CUtensorMap*>(pool->tmap), layer, static_cast<const __nv_bfloat16*>(q), qscale, rows);
  prof_end(pool, GB_PROF_GROUPED, s);
  pool->launches += 1;
  return cudaGetLastError();
}

cudaError_t launch_grouped(gb_pool* pool, int layer, const void* q, float scale, cudaStream_t s) {
  if (!pool->view.grouped || !pool->have_tmap) return cudaSuccess;
  switch (pool->view.G) {
    case 2: return launch_grouped_t<2>(pool, layer, q, scale, s);
    case 4: return launch_grouped_t<4>(pool, layer, q, scale, s);
    case 8: return launch_grouped_t<8>(pool, layer, q, scale, s);
  }
  return cudaErrorInvalidValue;
}

}  // namespace gb
