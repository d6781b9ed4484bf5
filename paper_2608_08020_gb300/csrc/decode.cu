// Split-KV flash-decode over the paged pool (per-beam path) and the LSE combine.
// Two per-beam kernels share the work decomposition and the record format below:
// k_decode_mma (bf16 pools with 128-dim heads; warp-level MMAs, further down) and
// k_decode (fp32 pools, and callers' own pages without a tensor map; paired fp32 FMAs).
//
// Work decomposition: the per-beam work of a step is the flat list of
// (beam, kv-head, 16-token chunk) units, ordered beam-major.  Every warp of a
// persistent grid takes one contiguous range of that list, so work is
// balanced to within one chunk whatever the beams' lengths.  A warp streams
// its chunks through a private ring of shared-memory stages filled by TMA.
// When its range leaves a (beam, head) it writes an unnormalised partial
// (m, l, o) for the G query heads of that KV head; the combine kernel merges
// the partials of each (beam, head) with the standard log-sum-exp rule.
//
// k_decode fills a stage with two 1D bulk copies (one 4 KiB K slab and one
// 4 KiB V slab per chunk, both contiguous in a page).  Its lane layout inside
// a warp: 4 token rows x 8 lanes.  Lane j of row r owns
// two 16-byte pieces of every token row (bytes [16j, 16j+16) and
// [128+16j, 128+16j+16) of the 256-byte row), i.e. 16 bf16 or 8 fp32 dims,
// and handles tokens r, r+4, r+8, r+12 of a chunk.  Scores are reduced with
// a 3-stage shuffle reduce-scatter inside each 8-lane row; softmax maxima
// are warp-wide so rescaling is a warp-uniform branch.
#include <cuda.h>
#include <cuda_bf16.h>
#include <math.h>

#include "decode_mma.cuh"
#include "internal.cuh"
#include "ptx.cuh"

namespace gb {

template <int DT>
struct KvTraits {
  static constexpr int ES = DT == GB_BF16 ? 2 : 4;
  static constexpr int D = DT == GB_BF16 ? 128 : 64;
  static constexpr int DPC = 16 / ES;  // dims per 16-byte piece
  static constexpr int DPL = 2 * DPC;  // dims per lane
  static constexpr int ROW_BYTES = D * ES;
  static constexpr int SLAB_BYTES = kChunk * ROW_BYTES;  // 4096
  static constexpr int STAGE_BYTES = 2 * SLAB_BYTES;     // K + V
  static_assert(ROW_BYTES == 256, "lane layout assumes 256-byte token rows");
};

// Unpack one 16-byte piece into DPC floats.
template <int DT>
__device__ __forceinline__ void unpack16(const uint4& u, float* f) {
  if constexpr (DT == GB_BF16) {
    const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      f[2 * k] = __uint_as_float(w[k] << 16);
      f[2 * k + 1] = __uint_as_float(w[k] & 0xffff0000u);
    }
  } else {
    f[0] = __uint_as_float(u.x);
    f[1] = __uint_as_float(u.y);
    f[2] = __uint_as_float(u.z);
    f[3] = __uint_as_float(u.w);
  }
}

template <int DT, int G>
struct DecodeSmem {
  using T = KvTraits<DT>;
  static constexpr int PBUF = kChunk * G * 4;
  // Rounded to 128 bytes so every warp's stages start 16-byte aligned (bulk-copy destinations).
  static constexpr int WARP_BYTES = (kDecodeStages * T::STAGE_BYTES + PBUF + 8 * kDecodeStages + 127) / 128 * 128;
  static_assert(WARP_BYTES % 128 == 0 && T::STAGE_BYTES % 16 == 0, "stage alignment");
  static constexpr int PLAN_BYTES = 3 * (kMaxBeams + 1) * 4;
  static constexpr int TOTAL = kDecodeWarps * WARP_BYTES + PLAN_BYTES;
};

// The same, as DPC / 2 pairs of consecutive dims (operands of the paired fp32 FMA).
template <int DT>
__device__ __forceinline__ void unpack16x2(const uint4& u, float2* f) {
  if constexpr (DT == GB_BF16) {
    const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
    for (int k = 0; k < 4; ++k) f[k] = make_float2(__uint_as_float(w[k] << 16), __uint_as_float(w[k] & 0xffff0000u));
  } else {
    f[0] = make_float2(__uint_as_float(u.x), __uint_as_float(u.y));
    f[1] = make_float2(__uint_as_float(u.z), __uint_as_float(u.w));
  }
}

template <int DT, int G>
__global__ void __launch_bounds__(kDecodeWarps * 32, 1)
    k_decode(PoolView v, int layer, const void* __restrict__ qptr, float qscale, int mode, int W) {
  pdl_wait();
  pdl_launch_dependents();
  using T = KvTraits<DT>;
  using S = DecodeSmem<DT, G>;
  constexpr int NS = G / 2;  // scores held per lane after the reduce-scatter
  constexpr int D = T::D, DPC = T::DPC, DPL = T::DPL;
  extern __shared__ __align__(128) unsigned char smem[];

  int* s_off = reinterpret_cast<int*>(smem + kDecodeWarps * S::WARP_BYTES);
  int* s_n = s_off + (kMaxBeams + 1);
  int* s_start = s_n + (kMaxBeams + 1);
  if (v.ctl[kCtlStepOk] == 0) return;
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
  const int row = lane >> 3, j = lane & 7;
  const int b0 = lane & 1, b1 = (lane >> 1) & 1, b2 = (lane >> 2) & 1;
  const int my_t = 4 * (2 * b2 + b1) + row;  // token (within the chunk) of this lane's scores
  unsigned char* wsm = smem + warp * S::WARP_BYTES;
  float* pbuf = reinterpret_cast<float*>(wsm + kDecodeStages * T::STAGE_BYTES);
  const uint32_t stage0 = smem_addr(wsm);
  const uint32_t bar0 = smem_addr(wsm + kDecodeStages * T::STAGE_BYTES + S::PBUF);

  const int Tot = s_off[v.max_beams];
  const int w = blockIdx.x * kDecodeWarps + warp;
  const int c = (Tot + W - 1) / W;
  const int x_begin = w * c;
  const int x_end = min(Tot, x_begin + c);
  if (x_begin >= x_end) return;

  if (lane == 0) {
    for (int s = 0; s < kDecodeStages; ++s) mbar_init(bar0 + 8 * s, 1);
    fence_mbar_init();
  }
  __syncwarp();

  // Locate the first chunk: the largest b with s_off[b] <= x_begin.
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
    const int r = x_begin - s_off[lo];
    it.h = r / it.n;
    it.i = r % it.n;
  }
  const uint64_t pol = policy_evict_first();
  // Page ids come from the block table 32 chunks at a time (lane l loads the page of chunk
  // i0 + l of the beam, one coalesced load) and are handed out by shuffles, so a chunk's
  // refill does not wait on a table load of its own.  Called by the whole warp.
  int pw_b = -1, pw_i0 = 0, pw_lane = 0;
  auto load_page = [&](const ChunkIter& q) -> int {
    if (q.b != pw_b || q.i < pw_i0 || q.i >= pw_i0 + 32) {
      pw_b = q.b;
      pw_i0 = q.i;
      const int i = pw_i0 + lane;
      pw_lane = i < q.n ? v.tables[(size_t)q.b * v.max_pages + (q.tok0 + i * kChunk) / v.P] : 0;
    }
    return __shfl_sync(0xffffffffu, pw_lane, q.i - pw_i0);
  };
  auto issue = [&](const ChunkIter& q, int page, int stage) {
    if (lane == 0) {
      if (page < 0 || page >= v.num_pages) {
        set_status(v.ctl, GB_ERR_INVALID);
        page = 0;
      }
      const int tok = q.tok0 + q.i * kChunk;
      const long long ek = kv_elem_offset(v, layer, page, 0, q.h, tok % v.P);
      const long long ev = kv_elem_offset(v, layer, page, 1, q.h, tok % v.P);
      const uint32_t bar = bar0 + 8 * stage;
      const uint32_t dst = stage0 + stage * T::STAGE_BYTES;
      mbar_arrive_expect_tx(bar, T::STAGE_BYTES);
      bulk_g2s(dst, v.kv + ek * T::ES, T::SLAB_BYTES, bar, pol);
      bulk_g2s(dst + T::SLAB_BYTES, v.kv + ev * T::ES, T::SLAB_BYTES, bar, pol);
    }
  };

  // Prologue: fill the ring.
  ChunkIter ip = it;
  int ip_x = x_begin;
  int ip_page = load_page(ip);
  for (int s = 0; s < kDecodeStages; ++s) {
    if (ip_x < x_end) {
      issue(ip, ip_page, s);
      ++ip_x;
      if (ip_x < x_end) {
        iter_advance(ip, s_n, s_start, v.Hkv, v.max_beams);
        ip_page = load_page(ip);
      }
    }
  }

  constexpr int DP2 = DPL / 2, DC2 = DPC / 2;  // dim pairs per lane / per 16-byte piece
  float2 qr[G][DP2];   // q (pre-scaled) and the accumulator as pairs of dims: every
  float2 o[G][DP2];    // multiply-add of Q.K and P.V is one paired fp32 FMA (FFMA2)
  float m_run[G];
  float l_lane[NS];
  int L = 0;
  bool fresh = true;
  const char* qbase = static_cast<const char*>(qptr);

  for (int x = x_begin, k = 0; x < x_end; ++x, ++k) {
    if (fresh) {
      // New (beam, head): load the G query rows for this lane's dims, pre-scaled.
      L = v.seq_len[it.b];
#pragma unroll
      for (int g = 0; g < G; ++g) {
        const char* qrow = qbase + ((size_t)(it.b * v.Hq + it.h * G + g) * D) * T::ES;
        const uint4 a = *reinterpret_cast<const uint4*>(qrow + 16 * j);
        const uint4 bq = *reinterpret_cast<const uint4*>(qrow + 128 + 16 * j);
        unpack16x2<DT>(a, qr[g]);
        unpack16x2<DT>(bq, qr[g] + DC2);
#pragma unroll
        for (int d = 0; d < DP2; ++d) {
          qr[g][d] = make_float2(qr[g][d].x * qscale, qr[g][d].y * qscale);
          o[g][d] = make_float2(0.f, 0.f);
        }
        m_run[g] = -INFINITY;
      }
#pragma unroll
      for (int kk = 0; kk < NS; ++kk) l_lane[kk] = 0.f;
      fresh = false;
    }
    const int stage = k % kDecodeStages;
    const uint32_t parity = (k / kDecodeStages) & 1;
    if (!mbar_wait_bounded(bar0 + 8 * stage, parity, kWaitLimitNs)) {
      if (lane == 0) set_status(v.ctl, GB_ERR_TIMEOUT);
      // Give copies still in flight a bounded chance to land before leaving.
      for (int s = 0; s < kDecodeStages; ++s) {
        const int kk = k + s;
        if (x + s < ip_x) mbar_wait_bounded(bar0 + 8 * (kk % kDecodeStages), (kk / kDecodeStages) & 1, kWaitLimitNs / 4);
      }
      return;
    }
    const unsigned char* Ks = wsm + stage * T::STAGE_BYTES;
    const unsigned char* Vs = Ks + T::SLAB_BYTES;
    const int tok0 = it.tok0 + it.i * kChunk;
    const bool partial = tok0 + kChunk > L;

    // ---- scores: 4 tokens per row, G heads each --------------------------
    float acc[4 * G];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const int t = 4 * i + row;
      const uint4 a = *reinterpret_cast<const uint4*>(Ks + t * T::ROW_BYTES + 16 * j);
      const uint4 bq = *reinterpret_cast<const uint4*>(Ks + t * T::ROW_BYTES + 128 + 16 * j);
      float2 kf[DP2];
      unpack16x2<DT>(a, kf);
      unpack16x2<DT>(bq, kf + DC2);
#pragma unroll
      for (int g = 0; g < G; ++g) {
        float2 sacc = make_float2(0.f, 0.f);
#pragma unroll
        for (int d = 0; d < DP2; ++d) sacc = __ffma2_rn(qr[g][d], kf[d], sacc);
        acc[i * G + g] = sacc.x + sacc.y;
      }
    }
    // Reduce-scatter over the 8 lanes of the row: 4G -> 2G -> G -> G/2 values.
#pragma unroll
    for (int kk = 0; kk < 2 * G; ++kk) {
      const bool up = lane & 4;
      const float keep = up ? acc[kk + 2 * G] : acc[kk];
      const float send = up ? acc[kk] : acc[kk + 2 * G];
      acc[kk] = keep + __shfl_xor_sync(0xffffffffu, send, 4);
    }
#pragma unroll
    for (int kk = 0; kk < G; ++kk) {
      const bool up = lane & 2;
      const float keep = up ? acc[kk + G] : acc[kk];
      const float send = up ? acc[kk] : acc[kk + G];
      acc[kk] = keep + __shfl_xor_sync(0xffffffffu, send, 2);
    }
    float sc[NS];
#pragma unroll
    for (int kk = 0; kk < NS; ++kk) {
      const bool up = lane & 1;
      const float keep = up ? acc[kk + NS] : acc[kk];
      const float send = up ? acc[kk] : acc[kk + NS];
      sc[kk] = keep + __shfl_xor_sync(0xffffffffu, send, 1);
      if (partial && tok0 + my_t >= L) sc[kk] = -INFINITY;
    }
    // ---- online softmax (warp-wide maxima, base 2) -------------------------
    float mx[NS], other[NS];
#pragma unroll
    for (int kk = 0; kk < NS; ++kk) {
      float m = sc[kk];
      m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, 2));
      m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, 4));
      m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, 8));
      m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, 16));
      mx[kk] = m;
    }
#pragma unroll
    for (int kk = 0; kk < NS; ++kk) other[kk] = __shfl_xor_sync(0xffffffffu, mx[kk], 1);
    bool grow = false;
    float m_new[G];
#pragma unroll
    for (int g = 0; g < G; ++g) {
      const float mc = ((g / NS) == b0) ? mx[g % NS] : other[g % NS];
      m_new[g] = fmaxf(m_run[g], mc);
      grow |= m_new[g] > m_run[g];
    }
    if (grow) {
      float alpha[G];
#pragma unroll
      for (int g = 0; g < G; ++g) {
        alpha[g] = exp2f(m_run[g] - m_new[g]);
        m_run[g] = m_new[g];
        const float2 a2 = make_float2(alpha[g], alpha[g]);
#pragma unroll
        for (int d = 0; d < DP2; ++d) o[g][d] = __fmul2_rn(o[g][d], a2);
      }
#pragma unroll
      for (int kk = 0; kk < NS; ++kk) l_lane[kk] *= b0 ? alpha[NS + kk] : alpha[kk];
    }
#pragma unroll
    for (int kk = 0; kk < NS; ++kk) {
      const float mr = b0 ? m_run[NS + kk] : m_run[kk];
      const float p = exp2f(sc[kk] - mr);
      l_lane[kk] += p;
      pbuf[my_t * G + NS * b0 + kk] = p;
    }
    __syncwarp();
    // ---- P.V -----------------------------------------------------------------
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const int t = 4 * i + row;
      float pv[G];
#pragma unroll
      for (int g = 0; g < G; ++g) pv[g] = pbuf[t * G + g];
      const uint4 a = *reinterpret_cast<const uint4*>(Vs + t * T::ROW_BYTES + 16 * j);
      const uint4 bq = *reinterpret_cast<const uint4*>(Vs + t * T::ROW_BYTES + 128 + 16 * j);
      float2 vf[DP2];
      unpack16x2<DT>(a, vf);
      unpack16x2<DT>(bq, vf + DC2);
      if (partial && tok0 + t >= L) {
#pragma unroll
        for (int d = 0; d < DP2; ++d) vf[d] = make_float2(0.f, 0.f);
      }
#pragma unroll
      for (int g = 0; g < G; ++g) {
        const float2 p2 = make_float2(pv[g], pv[g]);
#pragma unroll
        for (int d = 0; d < DP2; ++d) o[g][d] = __ffma2_rn(p2, vf[d], o[g][d]);
      }
    }
    __syncwarp();
    // The stage is free again: refill it with the chunk kDecodeStages ahead.
    if (ip_x < x_end) {
      if (lane == 0) fence_proxy_async_smem();
      issue(ip, ip_page, stage);
      ++ip_x;
      if (ip_x < x_end) {
        iter_advance(ip, s_n, s_start, v.Hkv, v.max_beams);
        ip_page = load_page(ip);
      }
    }
    // ---- end of this warp's share of (beam, head): write the partial --------
    const bool last_of_bh = (it.i == it.n - 1) || (x + 1 == x_end);
    if (last_of_bh) {
#pragma unroll
      for (int g = 0; g < G; ++g)
#pragma unroll
        for (int d = 0; d < DP2; ++d) {
          o[g][d].x += __shfl_xor_sync(0xffffffffu, o[g][d].x, 8);
          o[g][d].y += __shfl_xor_sync(0xffffffffu, o[g][d].y, 8);
          o[g][d].x += __shfl_xor_sync(0xffffffffu, o[g][d].x, 16);
          o[g][d].y += __shfl_xor_sync(0xffffffffu, o[g][d].y, 16);
        }
      float lsum[NS], lother[NS];
#pragma unroll
      for (int kk = 0; kk < NS; ++kk) {
        float s = l_lane[kk];
        s += __shfl_xor_sync(0xffffffffu, s, 2);
        s += __shfl_xor_sync(0xffffffffu, s, 4);
        s += __shfl_xor_sync(0xffffffffu, s, 8);
        s += __shfl_xor_sync(0xffffffffu, s, 16);
        lsum[kk] = s;
      }
#pragma unroll
      for (int kk = 0; kk < NS; ++kk) lother[kk] = __shfl_xor_sync(0xffffffffu, lsum[kk], 1);
      float* rec = v.partials + (size_t)(w + it.b * v.Hkv + it.h) * v.record_floats;
      if (row == 0) {
#pragma unroll
        for (int g = 0; g < G; ++g) {
          float* oa = rec + g * D + DPC * j;
          float* ob = rec + g * D + D / 2 + DPC * j;
#pragma unroll
          for (int e = 0; e < DC2; e += 2) {
            *reinterpret_cast<float4*>(oa + 2 * e) = make_float4(o[g][e].x, o[g][e].y, o[g][e + 1].x, o[g][e + 1].y);
            *reinterpret_cast<float4*>(ob + 2 * e) =
                make_float4(o[g][DC2 + e].x, o[g][DC2 + e].y, o[g][DC2 + e + 1].x, o[g][DC2 + e + 1].y);
          }
        }
      }
      if (lane == 0) {
#pragma unroll
        for (int g = 0; g < G; ++g) {
          rec[G * D + g] = m_run[g];
          rec[G * D + G + g] = ((g / NS) == b0) ? lsum[g % NS] : lother[g % NS];
        }
      }
      fresh = true;
    }
    if (x + 1 < x_end) iter_advance(it, s_n, s_start, v.Hkv, v.max_beams);
  }
}

// The per-beam kernel on its own (the per-beam path, every beam reading its whole context):
// every CTA of the grid takes part, and the pairs' records are merged into `out` in the same
// launch (combine.cuh).
template <int G>
__global__ void __launch_bounds__(kMmaWarps * 32, 1)
    k_decode_mma(PoolView v, const __grid_constant__ CUtensorMap tm, const __grid_constant__ CUtensorMap tmh,
                 int layer, const __nv_bfloat16* __restrict__ q, float qscale, int mode, float* __restrict__ out) {
  pdl_wait();
  pdl_launch_dependents();
  decode_mma_body<G>(v, &tm, &tmh, layer, q, qscale, mode, (int)blockIdx.x, (int)gridDim.x);
  combine_pairs<G>(v, mode, (int)gridDim.x * kMmaWarps, 0, false, (int)blockIdx.x, (int)gridDim.x, out);
}

// Merge the partial records of each (beam, kv head) into out[b][h*G+g][:]: the split-KV
// records of the warps that covered the beam's range (the log-sum-exp merge, base 2), after
// the fp32 kernel k_decode (the bf16 kernels merge their records themselves, combine.cuh).
// One CTA of 128 threads per (beam, kv head); thread t owns 4 consecutive output elements
// of one query head g and folds all records in one pass, 8 records of loads in flight at a
// time: M = running max of the records' m, acc = sum o * 2^(m - M), L = sum l * 2^(m - M),
// rescaled when M rises.  Every thread of a warp reads the same (m, l) words (one head per
// warp at D = 128, two at D = 64), so those loads are broadcasts; the o loads are float4
// and coalesced.
__global__ void __launch_bounds__(128) k_combine(PoolView v, int mode, int W, float* __restrict__ out) {
  pdl_wait();
  pdl_launch_dependents();
  const int bh = blockIdx.x;
  const int b = bh / v.Hkv, h = bh % v.Hkv;
  const int G = v.G, D = v.D, GD = G * D;
  float* ob = out + ((size_t)b * v.Hq + (size_t)h * G) * D;
  const bool ok = v.ctl[kCtlStepOk] != 0 && v.active[b] != 0;
  const int n = ok ? plan_n(v, mode)[b] : 0;
  if (n == 0) {
    for (int e = threadIdx.x; e < GD; e += blockDim.x) ob[e] = 0.f;
    return;
  }
  const int Tot = plan_off(v, mode)[v.max_beams];
  const int c = Tot > 0 ? (Tot + W - 1) / W : 1;
  const int off = plan_off(v, mode)[b] + h * n;
  const int first = off / c, npb = n > 0 ? (off + n - 1) / c - first + 1 : 0;  // per-beam records
  const int R = npb;
  const float* prec = v.partials + (size_t)(first + bh) * v.record_floats;
  auto rec_at = [&](int r) -> const float* { return prec + (size_t)r * v.record_floats; };
  const bool vec_out = (reinterpret_cast<uintptr_t>(ob) & 15) == 0;
  for (int e4 = threadIdx.x; e4 < GD / 4; e4 += blockDim.x) {
    const int g = (e4 * 4) / D;
    float M = -INFINITY, L = 0.f;
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
    for (int r0 = 0; r0 < R; r0 += 8) {
      float4 x[8];
      float mk[8], lk[8];
#pragma unroll
      for (int k = 0; k < 8; ++k) {
        const int r = r0 + k;
        if (r < R) {
          const float* rec = rec_at(r);
          x[k] = *reinterpret_cast<const float4*>(rec + 4 * e4);
          mk[k] = rec[GD + g];
          lk[k] = rec[GD + G + g];
        } else {
          x[k] = make_float4(0.f, 0.f, 0.f, 0.f);
          mk[k] = -INFINITY;  // a record that saw no token (or none at all) adds nothing
          lk[k] = 0.f;
        }
      }
      float mnew = M;
#pragma unroll
      for (int k = 0; k < 8; ++k) mnew = fmaxf(mnew, mk[k]);
      if (mnew == -INFINITY) continue;
      if (mnew > M) {  // M = -inf the first time: acc and L are still 0
        const float a = M == -INFINITY ? 0.f : exp2f(M - mnew);
        acc.x *= a;
        acc.y *= a;
        acc.z *= a;
        acc.w *= a;
        L *= a;
        M = mnew;
      }
#pragma unroll
      for (int k = 0; k < 8; ++k) {
        const float sc = mk[k] == -INFINITY ? 0.f : exp2f(mk[k] - M);
        acc.x = fmaf(x[k].x, sc, acc.x);
        acc.y = fmaf(x[k].y, sc, acc.y);
        acc.z = fmaf(x[k].z, sc, acc.z);
        acc.w = fmaf(x[k].w, sc, acc.w);
        L = fmaf(lk[k], sc, L);
      }
    }
    const float4 res = make_float4(acc.x / L, acc.y / L, acc.z / L, acc.w / L);
    if (vec_out) {
      *reinterpret_cast<float4*>(ob + 4 * e4) = res;
    } else {
      ob[4 * e4] = res.x;
      ob[4 * e4 + 1] = res.y;
      ob[4 * e4 + 2] = res.z;
      ob[4 * e4 + 3] = res.w;
    }
  }
}

template <int DT, int G>
static cudaError_t launch_decode_t(gb_pool* pool, int layer, const void* q, float scale, float* out, int mode,
                                   cudaStream_t s) {
  using S = DecodeSmem<DT, G>;
  const float qscale = scale * 1.4426950408889634f;  // log2(e): softmax in base 2
  cudaError_t e;
  if (DT == GB_BF16 && pool->have_dtmap && pool->num_sms * kMmaWarps <= kMaxDecodeWarps) {
    // One launch: the attention roles and the merge of their records.
    if (mode == 1) {
      e = launch_attention(pool, layer, q, scale, out, s);  // grouped and per-beam roles (grouped.cu)
    } else {
      e = set_max_dynamic_smem(reinterpret_cast<const void*>(k_decode_mma<G>), DecodeMmaSmem::TOTAL);
      if (e != cudaSuccess) return e;
      prof_begin(pool, GB_PROF_DECODE, s);
      e = launch_pdl(k_decode_mma<G>, pool->num_sms, kMmaWarps * 32, DecodeMmaSmem::TOTAL, s, pool->view,
                     *reinterpret_cast<const CUtensorMap*>(pool->dtmap),
                     *reinterpret_cast<const CUtensorMap*>(pool->dtmap_half), layer,
                     static_cast<const __nv_bfloat16*>(q), qscale, mode, out);
      prof_end(pool, GB_PROF_DECODE, s);
      pool->launches += 1;
    }
    prof_end(pool, GB_PROF_ATTENTION, s);
    return e;
  }
  if (mode == 1) return cudaErrorInvalidValue;  // a grouped pool always has the per-beam tensor maps
  const int W = pool->decode_warps;  // one CTA of kDecodeWarps warps per SM
  e = set_max_dynamic_smem(reinterpret_cast<const void*>(k_decode<DT, G>), S::TOTAL);
  if (e != cudaSuccess) return e;
  prof_begin(pool, GB_PROF_DECODE, s);
  e = launch_pdl(k_decode<DT, G>, W / kDecodeWarps, kDecodeWarps * 32, S::TOTAL, s, pool->view, layer, q, qscale,
                 mode, W);
  prof_end(pool, GB_PROF_DECODE, s);
  pool->launches += 1;
  if (e != cudaSuccess) return e;
  prof_end(pool, GB_PROF_ATTENTION, s);
  prof_begin(pool, GB_PROF_COMBINE, s);
  e = launch_pdl(k_combine, pool->view.max_beams * pool->view.Hkv, 128, 0, s, pool->view, mode, W, out);
  prof_end(pool, GB_PROF_COMBINE, s);
  pool->launches += 1;
  return e;
}

// One warp waits for the record count of pair 0 to reach one more than it holds; nothing
// raises it, so the wait runs out (the same bounded wait as the attention launch's merge).
__global__ void k_wait_selftest(PoolView v) {
  const int have = v.pair_cnt[0];
  if (!wait_pair_records(v, 0, have + 1, 0) && threadIdx.x == 0) set_status(v.ctl, GB_ERR_TIMEOUT);
}

cudaError_t launch_wait_selftest(gb_pool* pool, cudaStream_t s) {
  k_wait_selftest<<<1, 32, 0, s>>>(pool->view);
  return cudaGetLastError();
}

// Split-KV decode + combine on an explicit view (plan mode 0, W warps), for callers
// that supply their own tables and scratch instead of a pool.
template <int DT, int G>
static cudaError_t launch_view_t(const PoolView& v, int W, int layer, const void* q, float scale, float* out,
                                 cudaStream_t s) {
  using S = DecodeSmem<DT, G>;
  {
    const cudaError_t e = set_max_dynamic_smem(reinterpret_cast<const void*>(k_decode<DT, G>), S::TOTAL);
    if (e != cudaSuccess) return e;
  }
  const float qscale = scale * 1.4426950408889634f;
  k_decode<DT, G><<<W / kDecodeWarps, kDecodeWarps * 32, S::TOTAL, s>>>(v, layer, q, qscale, 0, W);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  k_combine<<<v.max_beams * v.Hkv, 128, 0, s>>>(v, 0, W, out);
  return cudaGetLastError();
}

cudaError_t launch_decode_view(const PoolView& v, int W, int layer, const void* q, float scale, float* out,
                               cudaStream_t s) {
  if (v.dtype == GB_BF16) {
    switch (v.G) {
      case 2: return launch_view_t<GB_BF16, 2>(v, W, layer, q, scale, out, s);
      case 4: return launch_view_t<GB_BF16, 4>(v, W, layer, q, scale, out, s);
      case 8: return launch_view_t<GB_BF16, 8>(v, W, layer, q, scale, out, s);
    }
  } else {
    switch (v.G) {
      case 2: return launch_view_t<GB_F32, 2>(v, W, layer, q, scale, out, s);
      case 4: return launch_view_t<GB_F32, 4>(v, W, layer, q, scale, out, s);
      case 8: return launch_view_t<GB_F32, 8>(v, W, layer, q, scale, out, s);
    }
  }
  return cudaErrorInvalidValue;
}

cudaError_t launch_decode(gb_pool* pool, int layer, const void* q, float scale, float* out, int mode,
                          cudaStream_t s) {
  const int G = pool->view.G;
  if (pool->view.dtype == GB_BF16) {
    switch (G) {
      case 2: return launch_decode_t<GB_BF16, 2>(pool, layer, q, scale, out, mode, s);
      case 4: return launch_decode_t<GB_BF16, 4>(pool, layer, q, scale, out, mode, s);
      case 8: return launch_decode_t<GB_BF16, 8>(pool, layer, q, scale, out, mode, s);
    }
  } else {
    switch (G) {
      case 2: return launch_decode_t<GB_F32, 2>(pool, layer, q, scale, out, mode, s);
      case 4: return launch_decode_t<GB_F32, 4>(pool, layer, q, scale, out, mode, s);
      case 8: return launch_decode_t<GB_F32, 8>(pool, layer, q, scale, out, mode, s);
    }
  }
  return cudaErrorInvalidValue;
}

}  // namespace gb
