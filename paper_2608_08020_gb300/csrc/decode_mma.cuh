// The per-beam split-KV work decomposition and the bf16 per-beam kernel body on warp-level
// MMAs, shared by decode.cu (the per-beam kernel) and grouped.cu (the one-launch attention
// kernel that runs the grouped and per-beam roles side by side).
#pragma once
#include <cuda.h>
#include <cuda_bf16.h>
#include <math.h>

#include "combine.cuh"
#include "internal.cuh"
#include "ptx.cuh"

namespace gb {

// Work decomposition: the per-beam work of a step is the flat list of (beam, kv-head, 16-token
// chunk) units, ordered beam-major; every warp takes one contiguous range of it.
struct ChunkIter {
  int b, h, i, n, tok0;
};

__device__ __forceinline__ void iter_advance(ChunkIter& it, const int* s_n, const int* s_start, int Hkv,
                                             int max_beams) {
  if (++it.i == it.n) {
    it.i = 0;
    if (++it.h == Hkv) {
      it.h = 0;
      do {
        ++it.b;
      } while (it.b < max_beams && s_n[it.b] == 0);
      if (it.b < max_beams) {
        it.n = s_n[it.b];
        it.tok0 = s_start[it.b];
      }
    }
  }
}

// ---- bf16 per-beam kernel on warp-level MMAs ---------------------------------
//
// The same work decomposition, ring and records as k_decode, for bf16 pools with 128-dim
// heads.  Staging: one 5D TMA per chunk brings K and V of the chunk's 16 tokens (8 KiB)
// with the 128-byte swizzle, laid out [8-token group][K|V][half of D][8 tokens][64 dims],
// so ldmatrix reads every 8x8 block without bank conflicts.  Arithmetic: m16n8k16 MMAs
// (bf16 in, fp32 accumulate), the G query heads of the KV head as the N = 8 columns
// (zero-padded):
//   S^T[16 tokens][8]  = K[16][128] . Q^T      8 MMAs, K by ldmatrix, Q^T held in registers
//   O^T[128][8]       += V^T[128][16] . P^T    8 MMAs, V^T by ldmatrix.trans
// P^T comes from S^T's accumulator fragments by two movmatrix transposes.  Lane (r, c) of
// the warp (r = lane / 4, c = lane % 4) holds the scores of query heads 2c and 2c + 1 for
// tokens r and r + 8, and exactly the O^T elements of the same two heads, so the softmax
// state and every rescale stay inside the lane.  Base-2 softmax; the running max is raised
// only when a chunk's max exceeds it by more than 8 (p <= 2^8 otherwise).  This cuts the
// per-chunk work of a warp from ~700 instructions per lane (k_decode's paired FMAs) to
// ~250-300 warp instructions, which is what bounds the per-beam kernel when it shares the
// GPU with the grouped kernel; 12 warps per SM with 2-stage rings hide more of each
// warp's instruction latency than 8 warps with 3 stages, in the same shared memory.
constexpr int kMmaStageBytes = 2 * kChunk * 128 * 2;  // K and V of 16 tokens x 128 bf16
#ifndef GB_MMA_STAGES
#define GB_MMA_STAGES 2  // ring depth per warp
#endif
#ifndef GB_MMA_CHAINS
#define GB_MMA_CHAINS 2  // independent accumulator chains of the 8 S^T MMAs of a chunk
#endif
constexpr int kMmaStages = GB_MMA_STAGES, kMmaChains = GB_MMA_CHAINS;
struct DecodeMmaSmem {
  static constexpr int STAGES = kMmaWarps * kMmaStages * kMmaStageBytes;
  static constexpr int BARS = kMmaWarps * kMmaStages * 8;
  static constexpr int PLAN_BYTES = 3 * (kMaxBeams + 1) * 4;
  static constexpr int TOTAL = 1024 + STAGES + BARS + PLAN_BYTES;  // 1024: alignment slack
  static_assert(TOTAL <= 232448, "shared memory per block");
};

// K and V of one 16-token chunk of one head: coordinates {0, 0, 0, 0, w}, w = the
// chunk's first K row / 8, box {64, 8, 2, 2, 2}.
__device__ __forceinline__ void tma_chunk(uint32_t dst, const CUtensorMap* tm, int w, uint32_t bar, uint64_t pol) {
  asm volatile(
      "cp.async.bulk.tensor.5d.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint"
      " [%0], [%1, {%2, %3, %4, %5, %6}], [%7], %8;" ::"r"(dst),
      "l"(tm), "r"(0), "r"(0), "r"(0), "r"(0), "r"(w), "r"(bar), "l"(pol)
      : "memory");
}

__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr)
               : "memory");
}

__device__ __forceinline__ void ldsm_x4_t(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr)
               : "memory");
}

// d += A[16x16] . B[16x8] (bf16 in, fp32 accumulate).
__device__ __forceinline__ void mma_bf16(float (&d)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3,
                                         uint32_t b0, uint32_t b1) {
  asm("mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, "
      "{%0, %1, %2, %3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

__device__ __forceinline__ uint32_t movmatrix_t(uint32_t x) {
  uint32_t y;
  asm("movmatrix.sync.aligned.m8n8.trans.b16 %0, %1;" : "=r"(y) : "r"(x));
  return y;
}

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  const __nv_bfloat162 t = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<const uint32_t*>(&t);
}

// The kernel's body, shared by the per-beam kernel (k_decode_mma, below in decode.cu) and the
// attention kernel that also runs the grouped role (k_attention, grouped.cu): this CTA is
// number `cta` of the `nctas` CTAs that take the per-beam work.  tm: 16-token boxes; tmh:
// 8-token boxes (the last chunk of a range when it holds at most 8 valid tokens).
template <int G>
__device__ __forceinline__ void decode_mma_body(const PoolView& v, const CUtensorMap* tm_p, const CUtensorMap* tmh_p,
                                                int layer, const __nv_bfloat16* __restrict__ q, float qscale,
                                                int mode, int cta, int nctas) {
  using S = DecodeMmaSmem;
  constexpr int D = 128;
  extern __shared__ __align__(1024) unsigned char smem_raw[];
  unsigned char* smem = smem_raw + ((1024 - (smem_addr(smem_raw) & 1023)) & 1023);
  int* s_off = reinterpret_cast<int*>(smem + S::STAGES + S::BARS);
  int* s_n = s_off + (kMaxBeams + 1);
  int* s_start = s_n + (kMaxBeams + 1);
  if (v.ctl[kCtlStepOk] == 0) return;
  const int W = nctas * kMmaWarps;  // warps that share the per-beam work
  {
    const int* off = plan_off(v, mode);
    const int* nn = plan_n(v, mode);
    const int* st = plan_start(v, mode);
    for (int i = threadIdx.x; i <= v.max_beams; i += blockDim.x) {
      s_off[i] = off[i];
      s_n[i] = i < v.max_beams ? nn[i] : 0;
      s_start[i] = i < v.max_beams ? st[i] : 0;
    }
  }
  __syncthreads();

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int r = lane >> 2, c = lane & 3;  // MMA fragment row (token / dim) and column pair (heads 2c, 2c + 1)
  const uint32_t stage0 = smem_addr(smem) + warp * kMmaStages * kMmaStageBytes;
  const uint32_t bar0 = smem_addr(smem) + S::STAGES + warp * kMmaStages * 8;

  const int Tot = s_off[v.max_beams];
  const int w = cta * kMmaWarps + warp;
  const int cw = (Tot + W - 1) / W;
  const int x_begin = w * cw;
  const int x_end = min(Tot, x_begin + cw);
  if (x_begin >= x_end) return;

  if (lane == 0) {
    for (int s = 0; s < kMmaStages; ++s) mbar_init(bar0 + 8 * s, 1);
    fence_mbar_init();
  }
  __syncwarp();

  ChunkIter it;
  {
    int lo = 0, hi = v.max_beams;  // invariant: s_off[lo] <= x < s_off[hi]
    while (hi - lo > 1) {
      const int mid = (lo + hi) >> 1;
      if (s_off[mid] <= x_begin) lo = mid; else hi = mid;
    }
    it.b = lo;
    it.n = s_n[lo];
    it.tok0 = s_start[lo];
    const int rr = x_begin - s_off[lo];
    it.h = rr / it.n;
    it.i = rr % it.n;
  }
  // L2 policy of the K/V chunks: evict first, as each is read once, unless this is the
  // per-beam path over a tree with shared pages, where siblings read the same pages again.
  const bool reread = mode == 0 && v.grouped && v.ctl[kCtlSegCount] > 0;
  const uint64_t pol = reread ? policy_evict_normal() : policy_evict_first();
  int pw_b = -1, pw_i0 = 0, pw_lane = 0;
  auto load_page = [&](const ChunkIter& qi) -> int {
    if (qi.b != pw_b || qi.i < pw_i0 || qi.i >= pw_i0 + 32) {
      pw_b = qi.b;
      pw_i0 = qi.i;
      const int i = pw_i0 + lane;
      pw_lane = i < qi.n ? v.tables[(size_t)qi.b * v.max_pages + (qi.tok0 + i * kChunk) / v.P] : 0;
    }
    return __shfl_sync(0xffffffffu, pw_lane, qi.i - pw_i0);
  };
  // Row group of a chunk's first K row: the whole pool has fewer than 2^31 rows (a condition
  // of the tensor map), so 32-bit arithmetic is exact; P is 16, 32 or 64.
  const int pg8 = v.P >> 3, layer_pages = layer * v.num_pages;
  auto issue = [&](const ChunkIter& qi, int page, int stage) {
    if (lane == 0) {
      if (page < 0 || page >= v.num_pages) {
        set_status(v.ctl, GB_ERR_INVALID);
        page = 0;
      }
      const int tok = qi.tok0 + qi.i * kChunk;
      const int wrow = ((layer_pages + page) * 2 * v.Hkv + qi.h) * pg8 + ((tok & (v.P - 1)) >> 3);
      const uint32_t bar = bar0 + 8 * stage;
      // The last chunk of a (beam, head) with at most 8 valid tokens brings only its first
      // 8-token group (the consumer masks the rest of the stage, whatever it holds).
      const bool half = qi.i == qi.n - 1 && v.seq_len[qi.b] - tok <= 8;
      mbar_arrive_expect_tx(bar, half ? kMmaStageBytes / 2 : kMmaStageBytes);
      tma_chunk(stage0 + stage * kMmaStageBytes, half ? tmh_p : tm_p, wrow, bar, pol);
    }
  };

  ChunkIter ip = it;
  int ip_x = x_begin;
  int ip_page = load_page(ip);
  for (int s = 0; s < kMmaStages; ++s) {
    if (ip_x < x_end) {
      issue(ip, ip_page, s);
      ++ip_x;
      if (ip_x < x_end) {
        iter_advance(ip, s_n, s_start, v.Hkv, v.max_beams);
        ip_page = load_page(ip);
      }
    }
  }

  // ldmatrix row addresses of this lane (lane = 8 * matrix + row).  K, non-transposed, for
  // S^T's A operand: matrix bit 0 picks the token half, bit 1 the 8-dim half of the
  // k-step.  V, transposed, for O^T's A operand: bit 0 picks the 8-dim half of the m-tile,
  // bit 1 the token half.  The 16-byte piece x of row y of a 1 KiB block sits at x ^ y.
  uint32_t koff[4], voff[4];
  {
    const int mi = lane >> 3, y = lane & 7;
#pragma unroll
    for (int jj = 0; jj < 4; ++jj) {
      koff[jj] = (mi & 1) * 4096 + y * 128 + (((2 * jj + (mi >> 1)) ^ y) << 4);
      voff[jj] = (mi >> 1) * 4096 + 2048 + y * 128 + (((2 * jj + (mi & 1)) ^ y) << 4);
    }
  }

  uint32_t qf[8][2];  // Q^T fragments: heads r < G, dims 16j + 2c (+1) and 16j + 8 + 2c (+1)
  float o[8][4];      // O^T fragments: dims 16mt + r (+8), heads 2c, 2c + 1
  float m0 = -INFINITY, m1 = -INFINITY, l0 = 0.f, l1 = 0.f;
  int L = 0;
  bool fresh = true;

  int stage = 0;
  uint32_t parity = 0;
  for (int x = x_begin, k = 0; x < x_end; ++x, ++k) {
    if (fresh) {
      L = v.seq_len[it.b];
      const uint32_t* qrow = reinterpret_cast<const uint32_t*>(q + ((size_t)it.b * v.Hq + it.h * G + r) * D);
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        qf[j][0] = r < G ? qrow[8 * j + c] : 0u;
        qf[j][1] = r < G ? qrow[8 * j + 4 + c] : 0u;
      }
#pragma unroll
      for (int mt = 0; mt < 8; ++mt) o[mt][0] = o[mt][1] = o[mt][2] = o[mt][3] = 0.f;
      m0 = m1 = -INFINITY;
      l0 = l1 = 0.f;
      fresh = false;
    }
    if (!mbar_wait_bounded(bar0 + 8 * stage, parity, kWaitLimitNs)) {
      if (lane == 0) set_status(v.ctl, GB_ERR_TIMEOUT);
      for (int s = 0; s < kMmaStages; ++s) {
        const int kk = k + s;
        if (x + s < ip_x) mbar_wait_bounded(bar0 + 8 * (kk % kMmaStages), (kk / kMmaStages) & 1, kWaitLimitNs / 4);
      }
      return;
    }
    const uint32_t sb = stage0 + stage * kMmaStageBytes;
    const int tok0 = it.tok0 + it.i * kChunk;
    const int nvalid = min(kChunk, L - tok0);  // >= 1: a chunk starts before the beam's length

    // ---- S^T = K . Q^T (kMmaChains independent accumulator chains) -----------
    float sacc[kMmaChains][4];
#pragma unroll
    for (int ch = 0; ch < kMmaChains; ++ch) sacc[ch][0] = sacc[ch][1] = sacc[ch][2] = sacc[ch][3] = 0.f;
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      uint32_t a0, a1, a2, a3;
      ldsm_x4(sb + koff[j & 3] + (j >> 2) * 1024, a0, a1, a2, a3);
      mma_bf16(sacc[j % kMmaChains], a0, a1, a2, a3, qf[j][0], qf[j][1]);
    }
    float sc[4];
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      float t = sacc[0][e];
#pragma unroll
      for (int ch = 1; ch < kMmaChains; ++ch) t += sacc[ch][e];
      sc[e] = t * qscale;
    }
    if (nvalid < kChunk) {
      // Tokens past the beam's length: no score, and zero V rows (the page's rows there
      // hold whatever the pool held), so that 0 * V stays 0 in the MMA.
      if (r >= nvalid) sc[0] = sc[1] = -INFINITY;
      if (r + 8 >= nvalid) sc[2] = sc[3] = -INFINITY;
      unsigned char* vs = smem + (sb - smem_addr(smem));
      for (int idx = lane; idx < (kChunk - nvalid) * 16; idx += 32) {
        const int t = nvalid + (idx >> 4), piece = idx & 15;
        *reinterpret_cast<uint4*>(vs + (t >> 3) * 4096 + 2048 + (piece >> 3) * 1024 + (t & 7) * 128 + (piece & 7) * 16) =
            make_uint4(0u, 0u, 0u, 0u);
      }
      fence_proxy_async_smem();  // ordered before the TMA that later refills this stage
      __syncwarp();
    }
    // ---- online softmax over the chunk's 16 tokens (per head column) ----------
    float mx0 = fmaxf(sc[0], sc[2]), mx1 = fmaxf(sc[1], sc[3]);
#pragma unroll
    for (int sh = 4; sh < 32; sh <<= 1) {
      mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, sh));
      mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, sh));
    }
    const bool up0 = mx0 > m0 + 8.f, up1 = mx1 > m1 + 8.f;
    if (__any_sync(0xffffffffu, up0 || up1)) {
      const float al0 = up0 ? ex2_approx(m0 - mx0) : 1.f;
      const float al1 = up1 ? ex2_approx(m1 - mx1) : 1.f;
      if (up0) m0 = mx0;
      if (up1) m1 = mx1;
#pragma unroll
      for (int mt = 0; mt < 8; ++mt) {
        o[mt][0] *= al0;
        o[mt][1] *= al1;
        o[mt][2] *= al0;
        o[mt][3] *= al1;
      }
      l0 *= al0;
      l1 *= al1;
    }
    const float p0 = ex2_approx(sc[0] - m0), p1 = ex2_approx(sc[1] - m1);
    const float p2 = ex2_approx(sc[2] - m0), p3 = ex2_approx(sc[3] - m1);
    l0 += p0 + p2;
    l1 += p1 + p3;
    const uint32_t pb0 = movmatrix_t(pack_bf16x2(p0, p1));  // P^T fragments: tokens 2c (+1), head r
    const uint32_t pb1 = movmatrix_t(pack_bf16x2(p2, p3));  // tokens 8 + 2c (+1)
    // ---- O^T += V^T . P^T ------------------------------------------------------
#pragma unroll
    for (int mt = 0; mt < 8; ++mt) {
      uint32_t a0, a1, a2, a3;
      ldsm_x4_t(sb + voff[mt & 3] + (mt >> 2) * 1024, a0, a1, a2, a3);
      mma_bf16(o[mt], a0, a1, a2, a3, pb0, pb1);
    }
    __syncwarp();
    if (ip_x < x_end) {
      if (lane == 0) fence_proxy_async_smem();
      issue(ip, ip_page, stage);
      ++ip_x;
      if (ip_x < x_end) {
        iter_advance(ip, s_n, s_start, v.Hkv, v.max_beams);
        ip_page = load_page(ip);
      }
    }
    if (++stage == kMmaStages) {
      stage = 0;
      parity ^= 1u;
    }
    const bool last_of_bh = (it.i == it.n - 1) || (x + 1 == x_end);
    if (last_of_bh) {
#pragma unroll
      for (int sh = 4; sh < 32; sh <<= 1) {
        l0 += __shfl_xor_sync(0xffffffffu, l0, sh);
        l1 += __shfl_xor_sync(0xffffffffu, l1, sh);
      }
      float* rec = v.partials + (size_t)(w + it.b * v.Hkv + it.h) * v.record_floats;
      if (2 * c < G) {
        float* o0 = rec + (2 * c) * D + r;
        float* o1 = o0 + D;
        const uint64_t rpol = policy_evict_last();  // the merge reads the record back from L2
#pragma unroll
        for (int mt = 0; mt < 8; ++mt) {
          st_hint(o0 + 16 * mt, o[mt][0], rpol);
          st_hint(o1 + 16 * mt, o[mt][1], rpol);
          st_hint(o0 + 16 * mt + 8, o[mt][2], rpol);
          st_hint(o1 + 16 * mt + 8, o[mt][3], rpol);
        }
        if (r == 0) {
          st_hint(rec + G * D + 2 * c, m0, rpol);
          st_hint(rec + G * D + 2 * c + 1, m1, rpol);
          st_hint(rec + G * D + G + 2 * c, l0, rpol);
          st_hint(rec + G * D + G + 2 * c + 1, l1, rpol);
        }
      }
      record_arrive(v, it.b * v.Hkv + it.h, lane);
      fresh = true;
    }
    if (x + 1 < x_end) iter_advance(it, s_n, s_start, v.Hkv, v.max_beams);
  }
  // Every chunk this warp issued has been consumed: its barriers' memory may serve again.
  if (lane == 0)
    for (int s = 0; s < kMmaStages; ++s) mbar_inval(bar0 + 8 * s);
}


}  // namespace gb
