// The history-aware sequence scorer (Appendix, "Evaluating Search Generalization",
// Eq. 4-6) run incrementally over the search: each thought step adds one position to
// every trace's step sequence, and the scorer's own key/value cache lives in a second
// beam pool (the step pool: one token per thought step), so a branched trace shares
// its parent's scorer history the way it shares its KV (forked block tables).
//
// Per step and layer, on the C slots of the step pool:
//   x_t  = GELU(W_in LN(h_t))                                   (Eq. 4)
//   u    = LN1(x);  q, k, v = W_qkv u, RoPE on q and k at the position t
//   a    = paged causal attention of q over the trace's cached k/v plus (k, v)
//          (gb_decode_attention on the step pool: it appends k, v first)
//   x   += W_o a;   u = LN2(x);   x += W_2 (SiLU(W_1 u) * W_3 u)  (Eq. 5)
//   y_t  = sigmoid(w_out . LN(x) + b_out)                        (Eq. 6)
// The matrix products are the split-K tcgen05 GEMM of gemm.cu (bf16 operands, fp32
// partials); each product's epilogue is one kernel that sums the partials in a fixed
// order and applies what follows it (GELU, residual add, the next LayerNorm, RoPE,
// SwiGLU, the output head), one CTA per row.  The residual stream x is fp32; the
// operands of the products (LayerNorm outputs, q/k/v, attention outputs, SwiGLU
// outputs) are rounded to bf16.
//
// Model shape: L = the step pool's layers, Hq query heads and Hkv key/value heads of
// 128 dims (the step pool's head counts, bf16 K/V), d_model = Hq * 128.  LayerNorm
// eps 1e-5; GELU the exact (erf) form; rotary pairs (i, i + 64) with angle
// t * 10000^(-i/64); softmax scale 1/sqrt(128).
#include "internal.cuh"

namespace gb {
namespace {

constexpr int kHd = 128;               // head dim of the scorer's attention
constexpr int kRowThreads = 256;       // epilogue CTAs: one per row
constexpr float kLnEps = 1e-5f;
constexpr int kPerLayer = 8;           // tensors per layer in the weight buffer
constexpr int kSplitBudget = 8;        // partial buffer: kSplitBudget x C x (widest product)

enum LayerTensor { kLn1G, kLn1B, kWqkv, kWo, kLn2G, kLn2B, kW13, kW2 };

struct Dims {
  int H, F, d, L, Hq, Hkv, G, Nqkv, C, Nmax, Umax;
};

size_t a256(size_t x) { return (x + 255) & ~size_t(255); }

bool make_dims(const gb_pool* p, const gb_scorer_config* cfg, Dims* s) {
  const gb_pool_config& c = p->cfg;
  if (!cfg || cfg->hidden_dim <= 0 || cfg->hidden_dim % 64 || cfg->ffn_dim <= 0 || cfg->ffn_dim % 64) return false;
  if (c.kv_dtype != GB_BF16 || c.head_dim != kHd) return false;
  s->H = cfg->hidden_dim;
  s->F = cfg->ffn_dim;
  s->L = c.num_layers;
  s->Hq = c.num_q_heads;
  s->Hkv = c.num_kv_heads;
  s->G = s->Hq / s->Hkv;
  s->d = s->Hq * kHd;
  s->Nqkv = (s->Hq + 2 * s->Hkv) * kHd;
  s->C = c.max_beams;
  s->Nmax = s->d > s->Nqkv ? s->d : s->Nqkv;
  s->Nmax = s->Nmax > 2 * s->F ? s->Nmax : 2 * s->F;
  s->Umax = s->H > s->d ? s->H : s->d;
  s->Umax = s->Umax > s->F ? s->Umax : s->F;
  return true;
}

int n_tensors(const Dims& s) { return 3 + kPerLayer * s.L + 4; }

// Byte sizes of the weight tensors in buffer order.
void tensor_sizes(const Dims& s, size_t* b) {
  int i = 0;
  b[i++] = 4 * (size_t)s.H;                 // ln_in gain
  b[i++] = 4 * (size_t)s.H;                 // ln_in bias
  b[i++] = 2 * (size_t)s.d * s.H;           // W_in [d][H]
  for (int l = 0; l < s.L; ++l) {
    b[i++] = 4 * (size_t)s.d;               // ln1 gain, bias
    b[i++] = 4 * (size_t)s.d;
    b[i++] = 2 * (size_t)s.Nqkv * s.d;      // W_qkv [(Hq + 2 Hkv) 128][d]: q heads, k heads, v heads
    b[i++] = 2 * (size_t)s.d * s.d;         // W_o [d][d]
    b[i++] = 4 * (size_t)s.d;               // ln2 gain, bias
    b[i++] = 4 * (size_t)s.d;
    b[i++] = 2 * (size_t)2 * s.F * s.d;     // W_13 [2F][d]: W_1 rows then W_3 rows
    b[i++] = 2 * (size_t)s.d * s.F;         // W_2 [d][F]
  }
  b[i++] = 4 * (size_t)s.d;                 // ln_out gain, bias
  b[i++] = 4 * (size_t)s.d;
  b[i++] = 4 * (size_t)s.d;                 // w_out
  b[i++] = 4;                               // b_out
}

size_t weight_offsets(const Dims& s, size_t* off) {
  size_t sz[3 + kPerLayer * 64 + 4];
  tensor_sizes(s, sz);
  size_t o = 0;
  for (int i = 0; i < n_tensors(s); ++i) {
    if (off) off[i] = o;
    o += a256(sz[i]);
  }
  return o;
}

struct Ws {
  size_t u, x, q, kn, vn, att, part, seedk, seedv, total;
  size_t part_floats;
};

Ws ws_layout(const Dims& s) {
  Ws w;
  size_t o = 0;
  auto take = [&](size_t bytes) {
    const size_t r = o;
    o += a256(bytes);
    return r;
  };
  w.u = take(2 * (size_t)s.C * s.Umax);
  w.x = take(4 * (size_t)s.C * s.d);
  w.q = take(2 * (size_t)s.C * s.d);
  w.kn = take(2 * (size_t)s.C * s.Hkv * kHd);
  w.vn = take(2 * (size_t)s.C * s.Hkv * kHd);
  w.att = take(4 * (size_t)s.C * s.d);
  w.part_floats = (size_t)kSplitBudget * s.C * s.Nmax;
  w.part = take(4 * w.part_floats);
  w.seedk = take(2 * (size_t)s.L * s.Hkv * kHd);
  w.seedv = take(2 * (size_t)s.L * s.Hkv * kHd);
  w.total = o;
  return w;
}

// Fixed-order block sum (xor butterfly in each warp, then the warps in order); every
// thread gets the total.  `red` holds 33 floats.
__device__ __forceinline__ float block_sum(float v, float* red) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  if (lane == 0) red[warp] = v;
  __syncthreads();
  if (threadIdx.x == 0) {
    float t = 0.f;
    for (int w = 0; w < (int)(blockDim.x >> 5); ++w) t += red[w];
    red[32] = t;
  }
  __syncthreads();
  const float t = red[32];
  __syncthreads();
  return t;
}

// LayerNorm of the row held in shared memory (n floats): gain and bias applied, bf16 out.
__device__ void layer_norm_row(const float* row, int n, const float* __restrict__ g, const float* __restrict__ b,
                               __nv_bfloat16* __restrict__ out, float* red) {
  float s = 0.f;
  for (int i = threadIdx.x; i < n; i += blockDim.x) s += row[i];
  const float mu = block_sum(s, red) / (float)n;
  float v = 0.f;
  for (int i = threadIdx.x; i < n; i += blockDim.x) {
    const float c = row[i] - mu;
    v = fmaf(c, c, v);
  }
  const float var = block_sum(v, red) / (float)n;
  const float r = 1.0f / sqrtf(var + kLnEps);
  for (int i = threadIdx.x; i < n; i += blockDim.x) out[i] = __float2bfloat16_rn((row[i] - mu) * r * g[i] + b[i]);
}

__device__ __forceinline__ float sum_partials(const float* __restrict__ P, int splits, int M, int N, int m, int n) {
  float z = 0.f;
  for (int k = 0; k < splits; ++k) z += P[((size_t)k * M + m) * N + n];
  return z;
}

__device__ __forceinline__ bool row_live(const int* active, int m) { return active == nullptr || active[m] != 0; }

// Input LayerNorm of Eq. 4: u[m] = LN_in(h[m]) (bf16 h, H wide, H % 64 == 0).  Inactive
// rows give zeros.  16-byte loads and stores (8 values); the row is staged in shared memory.
__global__ void __launch_bounds__(kRowThreads) k_ln_in(const __nv_bfloat16* __restrict__ h, int H,
                                                       const float* __restrict__ g, const float* __restrict__ b,
                                                       const int* __restrict__ active,
                                                       __nv_bfloat16* __restrict__ u) {
  pdl_wait();
  pdl_launch_dependents();
  extern __shared__ float row[];
  __shared__ float red[33];
  const int m = blockIdx.x, nv = H / 8;
  uint4* out = reinterpret_cast<uint4*>(u + (size_t)m * H);
  if (!row_live(active, m)) {
    for (int i = threadIdx.x; i < nv; i += blockDim.x) out[i] = make_uint4(0, 0, 0, 0);
    return;
  }
  const uint4* in = reinterpret_cast<const uint4*>(h + (size_t)m * H);
  float s = 0.f;
  for (int i = threadIdx.x; i < nv; i += blockDim.x) {
    const uint4 q = in[i];
    const __nv_bfloat162* p2 = reinterpret_cast<const __nv_bfloat162*>(&q);
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const float2 f = __bfloat1622float2(p2[j]);
      row[8 * i + 2 * j] = f.x;
      row[8 * i + 2 * j + 1] = f.y;
      s += f.x + f.y;
    }
  }
  const float mu = block_sum(s, red) / (float)H;
  float v = 0.f;
  for (int i = threadIdx.x; i < H; i += blockDim.x) {
    const float c = row[i] - mu;
    v = fmaf(c, c, v);
  }
  const float r = 1.0f / sqrtf(block_sum(v, red) / (float)H + kLnEps);
  for (int i = threadIdx.x; i < nv; i += blockDim.x) {
    uint4 q;
    __nv_bfloat162* p2 = reinterpret_cast<__nv_bfloat162*>(&q);
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int e = 8 * i + 2 * j;
      p2[j] = __floats2bfloat162_rn((row[e] - mu) * r * g[e] + b[e], (row[e + 1] - mu) * r * g[e + 1] + b[e + 1]);
    }
    out[i] = q;
  }
}

enum RowMode { kGeluLn = 0, kResidLn = 1, kResidHead = 2 };

// Epilogue of a d-wide product, one CTA per row m:
//   kGeluLn:    x[m] = GELU(z)            then u[m] = LN(x[m])           (Eq. 4, then LN1 of layer 0)
//   kResidLn:   x[m] += z                 then u[m] = LN(x[m])           (residual, then the next LN)
//   kResidHead: x[m] += z                 then score[m] = sigmoid(w_out . LN(x[m]) + b_out)   (Eq. 6)
// z = the sum of the product's K-split partials.  Inactive rows: u = 0, score = 0.
template <int Mode>
__global__ void __launch_bounds__(kRowThreads) k_row_epilogue(const float* __restrict__ P, int splits, int M, int d,
                                                              float* __restrict__ x, const float* __restrict__ g,
                                                              const float* __restrict__ b, const int* __restrict__ active,
                                                              __nv_bfloat16* __restrict__ u,
                                                              const float* __restrict__ w_out,
                                                              const float* __restrict__ b_out,
                                                              float* __restrict__ score) {
  pdl_wait();
  pdl_launch_dependents();
  extern __shared__ float row[];
  __shared__ float red[33];
  const int m = blockIdx.x;
  if (!row_live(active, m)) {
    if (Mode == kResidHead) {
      if (score && threadIdx.x == 0) score[m] = 0.f;
    } else {
      for (int i = threadIdx.x; i < d; i += blockDim.x) u[(size_t)m * d + i] = __float2bfloat16_rn(0.f);
    }
    return;
  }
  float* xm = x + (size_t)m * d;
  for (int i = threadIdx.x; i < d; i += blockDim.x) {
    const float z = sum_partials(P, splits, M, d, m, i);
    const float y = Mode == kGeluLn ? 0.5f * z * (1.0f + erff(z * 0.70710678118654752f)) : xm[i] + z;
    xm[i] = y;
    row[i] = y;
  }
  __syncthreads();
  if (Mode != kResidHead) {
    layer_norm_row(row, d, g, b, u + (size_t)m * d, red);
    return;
  }
  // Output head: LN, dot with w_out (fixed order), bias, sigmoid.
  float s = 0.f;
  for (int i = threadIdx.x; i < d; i += blockDim.x) s += row[i];
  const float mu = block_sum(s, red) / (float)d;
  float v = 0.f;
  for (int i = threadIdx.x; i < d; i += blockDim.x) {
    const float c = row[i] - mu;
    v = fmaf(c, c, v);
  }
  const float r = 1.0f / sqrtf(block_sum(v, red) / (float)d + kLnEps);
  float dot = 0.f;
  for (int i = threadIdx.x; i < d; i += blockDim.x) dot = fmaf((row[i] - mu) * r * g[i] + b[i], w_out[i], dot);
  const float y = block_sum(dot, red) + b_out[0];
  if (threadIdx.x == 0 && score) score[m] = 1.0f / (1.0f + expf(-y));
}

// Epilogue of the q/k/v product, one CTA per row m: sums the partials, rotates the
// (i, i + 64) pairs of every q and k head by pos * 10000^(-i/64) with pos = pos_of[m] +
// pos_shift (0 without pos_of), and writes q [M][Hq][128], k and v [M][Hkv][128] in bf16.
__global__ void __launch_bounds__(kRowThreads) k_qkv_epilogue(const float* __restrict__ P, int splits, int M, int Hq,
                                                              int Hkv, const int* __restrict__ pos_of, int pos_shift,
                                                              const int* __restrict__ active,
                                                              __nv_bfloat16* __restrict__ q,
                                                              __nv_bfloat16* __restrict__ kn,
                                                              __nv_bfloat16* __restrict__ vn) {
  pdl_wait();
  pdl_launch_dependents();
  const int m = blockIdx.x;
  const int N = (Hq + 2 * Hkv) * kHd;
  const bool live = row_live(active, m);
  const float pos = pos_of && live ? (float)(pos_of[m] + pos_shift) : 0.f;
  const int pairs = (Hq + Hkv) * (kHd / 2);
  for (int j = threadIdx.x; j < pairs; j += blockDim.x) {
    const int head = j / (kHd / 2), i = j % (kHd / 2);
    const int col = head * kHd + i;
    float a = 0.f, c = 0.f;
    if (live) {
      const float x1 = sum_partials(P, splits, M, N, m, col), x2 = sum_partials(P, splits, M, N, m, col + kHd / 2);
      const float ang = pos * powf(10000.0f, -(float)i / (float)(kHd / 2));
      float sn, cs;
      sincosf(ang, &sn, &cs);
      a = x1 * cs - x2 * sn;
      c = x1 * sn + x2 * cs;
    }
    __nv_bfloat16* dst = head < Hq ? q + ((size_t)m * Hq + head) * kHd : kn + ((size_t)m * Hkv + head - Hq) * kHd;
    dst[i] = __float2bfloat16_rn(a);
    dst[i + kHd / 2] = __float2bfloat16_rn(c);
  }
  for (int j = threadIdx.x; j < Hkv * kHd; j += blockDim.x)
    vn[(size_t)m * Hkv * kHd + j] =
        __float2bfloat16_rn(live ? sum_partials(P, splits, M, N, m, (Hq + Hkv) * kHd + j) : 0.f);
}

// SwiGLU epilogue: u[m][n] = SiLU(z[m][n]) * z[m][F + n] in bf16 (z = W_13 u, F wide halves).
__global__ void __launch_bounds__(kRowThreads) k_swiglu_epilogue(const float* __restrict__ P, int splits, int M, int F,
                                                                 const int* __restrict__ active,
                                                                 __nv_bfloat16* __restrict__ u) {
  pdl_wait();
  pdl_launch_dependents();
  const int m = blockIdx.x;
  const bool live = row_live(active, m);
  for (int n = threadIdx.x; n < F; n += blockDim.x) {
    float y = 0.f;
    if (live) {
      const float g1 = sum_partials(P, splits, M, 2 * F, m, n), g3 = sum_partials(P, splits, M, 2 * F, m, F + n);
      y = g1 / (1.0f + expf(-g1)) * g3;
    }
    u[(size_t)m * F + n] = __float2bfloat16_rn(y);
  }
}

// Attention outputs (fp32) to the bf16 operand of W_o.
__global__ void k_to_bf16(const float* __restrict__ a, size_t n, __nv_bfloat16* __restrict__ u) {
  pdl_wait();
  pdl_launch_dependents();
  for (size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x; i < n; i += (size_t)gridDim.x * blockDim.x)
    u[i] = __float2bfloat16_rn(a[i]);
}

// Attention of the first position alone (the seed row): softmax over one key is 1, so
// query head h returns the value of KV head h / G.
__global__ void k_first_position_attention(const __nv_bfloat16* __restrict__ vn, int Hq, int G,
                                           __nv_bfloat16* __restrict__ u) {
  pdl_wait();
  pdl_launch_dependents();
  for (int j = threadIdx.x; j < Hq * kHd; j += blockDim.x) u[j] = vn[(j / kHd / G) * kHd + j % kHd];
}

struct Run {
  gb_pool* pool;
  Dims s;
  const char* w;
  size_t off[3 + kPerLayer * 64 + 4];
  char* ws;
  Ws L;
  cudaStream_t st;
  int launches = 0;

  template <class T>
  const T* wt(int i) const { return reinterpret_cast<const T*>(w + off[i]); }
  int layer_tensor(int l, int t) const { return 3 + kPerLayer * l + t; }
  int tail(int t) const { return 3 + kPerLayer * s.L + t; }
  __nv_bfloat16* u() const { return reinterpret_cast<__nv_bfloat16*>(ws + L.u); }
  float* x() const { return reinterpret_cast<float*>(ws + L.x); }
  float* part() const { return reinterpret_cast<float*>(ws + L.part); }

  // P = A [M][K] . B [N][K]^T as K-split partials; returns the split count (0 on failure).
  int gemm(const void* A, int M, const void* B, int N, int K) {
    const int splits = gemm_splits(M, N, K, pool->num_sms, L.part_floats);
    if (splits == 0) return 0;
    if (gemm_partials(A, M, B, N, K, splits, part(), pool->view.ctl, st) != cudaSuccess) return 0;
    ++launches;
    return splits;
  }

  template <int Mode>
  void rows(int splits, int M, const float* g, const float* b, const int* active, const float* w_out,
            const float* b_out, float* score) {
    launch_pdl(k_row_epilogue<Mode>, M, kRowThreads, s.d * sizeof(float), st, part(), splits, M, s.d, x(), g, b,
               active, u(), w_out, b_out, score);
    ++launches;
  }

  // The layer stack on M rows.  step = true: rows are the step pool's slots, attention
  // runs over each trace's cached history (and appends to it); RoPE positions are the
  // slots' sequence lengths.  step = false: one row at position 0 (the seed), whose
  // per-layer k and v go to the seed buffers.
  bool layers(int M, bool step, const int* active, float* score) {
    const int* pos_of = step ? pool->view.seq_len : nullptr;
    for (int l = 0; l < s.L; ++l) {
      int sp = gemm(u(), M, wt<__nv_bfloat16>(layer_tensor(l, kWqkv)), s.Nqkv, s.d);
      if (!sp) return false;
      __nv_bfloat16* q = reinterpret_cast<__nv_bfloat16*>(ws + L.q);
      __nv_bfloat16* kn = reinterpret_cast<__nv_bfloat16*>(ws + (step ? L.kn : L.seedk)) +
                          (step ? 0 : (size_t)l * s.Hkv * kHd);
      __nv_bfloat16* vn = reinterpret_cast<__nv_bfloat16*>(ws + (step ? L.vn : L.seedv)) +
                          (step ? 0 : (size_t)l * s.Hkv * kHd);
      // Layer 0 opens the step pool's step, which advances every length by one: the new
      // position is seq_len before layer 0 and seq_len - 1 after it.
      launch_pdl(k_qkv_epilogue, M, kRowThreads, 0, st, part(), sp, M, s.Hq, s.Hkv, pos_of, l > 0 ? -1 : 0, active,
                 q, kn, vn);
      ++launches;
      if (!step && l + 1 == s.L) break;  // the seed needs only each layer's k and v
      if (step) {
        float* att = reinterpret_cast<float*>(ws + L.att);
        if (gb_decode_attention(pool, l, q, kn, vn, 0.08838834764831845f, att, GB_PATH_AUTO,
                                reinterpret_cast<gb_stream_t>(st)) != GB_OK)
          return false;
        const size_t n = (size_t)M * s.d;
        launch_pdl(k_to_bf16, (int)((n + 255) / 256 < 4096 ? (n + 255) / 256 : 4096), 256, 0, st,
                   static_cast<const float*>(att), n, u());
      } else {
        k_first_position_attention<<<1, kRowThreads, 0, st>>>(vn, s.Hq, s.G, u());
      }
      ++launches;
      sp = gemm(u(), M, wt<__nv_bfloat16>(layer_tensor(l, kWo)), s.d, s.d);
      if (!sp) return false;
      rows<kResidLn>(sp, M, wt<float>(layer_tensor(l, kLn2G)), wt<float>(layer_tensor(l, kLn2B)), active, nullptr,
                     nullptr, nullptr);
      sp = gemm(u(), M, wt<__nv_bfloat16>(layer_tensor(l, kW13)), 2 * s.F, s.d);
      if (!sp) return false;
      launch_pdl(k_swiglu_epilogue, M, kRowThreads, 0, st, part(), sp, M, s.F, active, u());
      ++launches;
      sp = gemm(u(), M, wt<__nv_bfloat16>(layer_tensor(l, kW2)), s.d, s.F);
      if (!sp) return false;
      if (l + 1 < s.L)
        rows<kResidLn>(sp, M, wt<float>(layer_tensor(l + 1, kLn1G)), wt<float>(layer_tensor(l + 1, kLn1B)), active,
                       nullptr, nullptr, nullptr);
      else if (step)
        rows<kResidHead>(sp, M, wt<float>(tail(0)), wt<float>(tail(1)), active, wt<float>(tail(2)),
                         wt<float>(tail(3)), score);
    }
    return true;
  }

  // Eq. 4 and LN1 of layer 0 on M rows of h.
  bool input(const void* h, int M, const int* active) {
    launch_pdl(k_ln_in, M, kRowThreads, s.H * sizeof(float), st, reinterpret_cast<const __nv_bfloat16*>(h), s.H,
               wt<float>(0), wt<float>(1), active, u());
    ++launches;
    const int sp = gemm(u(), M, wt<__nv_bfloat16>(2), s.d, s.H);
    if (!sp) return false;
    rows<kGeluLn>(sp, M, wt<float>(layer_tensor(0, kLn1G)), wt<float>(layer_tensor(0, kLn1B)), active, nullptr,
                  nullptr, nullptr);
    return true;
  }
};

gb_status prepare(gb_pool* pool, const gb_scorer_config* cfg, const void* weights, void* ws, gb_stream_t stream,
                  Run* r) {
  if (!pool) return GB_ERR_INVALID;
  if (!make_dims(pool, cfg, &r->s)) return fail(pool, GB_ERR_UNSUPPORTED, "scorer: needs a bf16 step pool with 128-dim heads and sizes in multiples of 64");
  if (r->s.L > 64) return fail(pool, GB_ERR_UNSUPPORTED, "scorer: at most 64 layers");
  if (!weights || !ws || ((uintptr_t)weights & 255) || ((uintptr_t)ws & 255))
    return fail(pool, GB_ERR_INVALID, "scorer: weights and workspace must be 256-byte aligned device buffers");
  if (r->s.d * sizeof(float) > 48 * 1024 || r->s.H * sizeof(float) > 48 * 1024)
    return fail(pool, GB_ERR_UNSUPPORTED, "scorer: hidden_dim and d_model up to 12288");
  if (pool->next_layer != 0) return fail(pool, GB_ERR_STATE, "scorer: step pool has an open step");
  r->pool = pool;
  r->w = reinterpret_cast<const char*>(weights);
  weight_offsets(r->s, r->off);
  r->ws = reinterpret_cast<char*>(ws);
  r->L = ws_layout(r->s);
  r->st = reinterpret_cast<cudaStream_t>(stream);
  return GB_OK;
}

}  // namespace
}  // namespace gb

using namespace gb;

extern "C" gb_status gb_scorer_sizes(gb_pool* step_pool, const gb_scorer_config* cfg, size_t* weight_bytes,
                                     size_t* workspace_bytes, size_t* offsets, int max_offsets, int* n_offsets) {
  if (!step_pool) return GB_ERR_INVALID;
  Dims s;
  if (!make_dims(step_pool, cfg, &s)) return fail(step_pool, GB_ERR_UNSUPPORTED, "scorer: unsupported shape");
  if (s.L > 64) return fail(step_pool, GB_ERR_UNSUPPORTED, "scorer: at most 64 layers");
  size_t off[3 + kPerLayer * 64 + 4];
  const size_t wb = weight_offsets(s, off);
  if (weight_bytes) *weight_bytes = wb;
  if (workspace_bytes) *workspace_bytes = ws_layout(s).total;
  if (n_offsets) *n_offsets = n_tensors(s);
  if (offsets) {
    if (max_offsets < n_tensors(s)) return fail(step_pool, GB_ERR_INVALID, "scorer: offsets array too short");
    for (int i = 0; i < n_tensors(s); ++i) offsets[i] = off[i];
  }
  return GB_OK;
}

extern "C" gb_status gb_scorer_seed(gb_pool* step_pool, const gb_scorer_config* cfg, const void* weights_dev,
                                    void* workspace_dev, const void* h0_dev, int n_beams, gb_stream_t stream) {
  Run r;
  gb_status st = prepare(step_pool, cfg, weights_dev, workspace_dev, stream, &r);
  if (st != GB_OK) return st;
  if (!h0_dev || ((uintptr_t)h0_dev & 15)) return fail(step_pool, GB_ERR_INVALID, "scorer_seed: h0 must be 16-byte aligned");
  if (step_pool->seeded) return fail(step_pool, GB_ERR_STATE, "scorer_seed: step pool already seeded");
  if (n_beams < 1 || n_beams > r.s.C) return fail(step_pool, GB_ERR_INVALID, "scorer_seed: bad beam count");
  const bool ok = r.input(h0_dev, 1, nullptr) && r.layers(1, false, nullptr, nullptr);
  step_pool->launches += r.launches;
  st = check_launch(step_pool, "scorer_seed");
  if (st != GB_OK) return st;
  if (!ok) return fail(step_pool, GB_ERR_CUDA, "scorer_seed: a launch failed");
  return gb_pool_seed(step_pool, n_beams, 1, r.ws + r.L.seedk, r.ws + r.L.seedv, stream);
}

extern "C" gb_status gb_scorer_step(gb_pool* step_pool, const gb_scorer_config* cfg, const void* weights_dev,
                                    void* workspace_dev, const void* hidden_dev, float* score_out_dev,
                                    gb_stream_t stream) {
  Run r;
  gb_status st = prepare(step_pool, cfg, weights_dev, workspace_dev, stream, &r);
  if (st != GB_OK) return st;
  if (!hidden_dev || ((uintptr_t)hidden_dev & 15) || !score_out_dev)
    return fail(step_pool, GB_ERR_INVALID, "scorer_step: hidden (16-byte aligned) and score_out required");
  if (!step_pool->seeded) return fail(step_pool, GB_ERR_STATE, "scorer_step: step pool not seeded");
  const int* active = step_pool->view.active;
  prof_begin(step_pool, GB_PROF_PROBE, r.st);
  const bool ok = r.input(hidden_dev, r.s.C, active) && r.layers(r.s.C, true, active, score_out_dev);
  if (ok) prof_end(step_pool, GB_PROF_PROBE, r.st);
  step_pool->launches += r.launches;
  st = check_launch(step_pool, "scorer_step");
  if (st != GB_OK) return st;
  return ok ? GB_OK : fail(step_pool, GB_ERR_CUDA, "scorer_step: a launch failed");
}
