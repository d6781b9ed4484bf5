// Seeded, counter-based input generator on the device.  Bit-identical to
// workload/gen.py (same SplitMix64 finaliser, stream keys, Irwin-Hall(4)
// normal approximation and fp32/bf16 rounding); see that file for the
// definition.  It holds none of the beam-search arithmetic and is used only to
// produce large synthetic inputs in device memory.
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace {

constexpr uint64_t kGamma = 0x9E3779B97F4A7C15ull;

__device__ __forceinline__ uint64_t mix64(uint64_t z) {
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

struct Field {
  long long base, c0, c1;  // value = base + c0 * i0 + c1 * i1 (taken mod 2^64)
};

struct GenArgs {
  void* out;
  int dtype;  // 0 fp32, 1 bf16
  int n0, n1, n2;
  int nfields;
  Field f[6];
  float scale;
  const float* row_scale;  // optional, indexed by j / row_scale_div
  int row_scale_div;
};

__global__ void k_gen_normal(GenArgs a) {
  const long long total = (long long)a.n0 * a.n1 * a.n2;
  for (long long e = blockIdx.x * (long long)blockDim.x + threadIdx.x; e < total;
       e += (long long)gridDim.x * blockDim.x) {
    const int j = (int)(e % a.n2);
    const long long r = e / a.n2;
    const int i1 = (int)(r % a.n1);
    const int i0 = (int)(r / a.n1);
    uint64_t h = 0;
    for (int k = 0; k < a.nfields; ++k) {
      const uint64_t fv = (uint64_t)a.f[k].base + (uint64_t)a.f[k].c0 * (uint64_t)i0 + (uint64_t)a.f[k].c1 * (uint64_t)i1;
      h = mix64((h + kGamma) ^ fv);
    }
    const uint64_t bits = mix64(h + (uint64_t)(j + 1) * kGamma);
    const uint32_t s = (uint32_t)(bits & 0xffffu) + (uint32_t)((bits >> 16) & 0xffffu) +
                       (uint32_t)((bits >> 32) & 0xffffu) + (uint32_t)(bits >> 48);
    float x = __fmul_rn((float)((int)s - 131070), __uint_as_float(0x37DDB3D7u));
    if (a.scale != 1.0f) x = __fmul_rn(x, a.scale);
    if (a.row_scale) x = __fmul_rn(x, a.row_scale[j / a.row_scale_div]);
    if (a.dtype == 1)
      static_cast<__nv_bfloat16*>(a.out)[e] = __float2bfloat16_rn(x);
    else
      static_cast<float*>(a.out)[e] = x;
  }
}

}  // namespace

// fields: nfields triples (base, c0, c1).  Returns a cudaError_t value.
extern "C" int gbgen_normal(void* out, int dtype, int n0, int n1, int n2, int nfields, const long long* fields,
                            float scale, const float* row_scale_dev, int row_scale_div, void* stream) {
  if (nfields < 0 || nfields > 6 || n0 < 0 || n1 < 0 || n2 < 0) return (int)cudaErrorInvalidValue;
  GenArgs a{};
  a.out = out;
  a.dtype = dtype;
  a.n0 = n0;
  a.n1 = n1;
  a.n2 = n2;
  a.nfields = nfields;
  for (int k = 0; k < nfields; ++k) a.f[k] = Field{fields[3 * k], fields[3 * k + 1], fields[3 * k + 2]};
  a.scale = scale;
  a.row_scale = row_scale_dev;
  a.row_scale_div = row_scale_div > 0 ? row_scale_div : 1;
  const long long total = (long long)n0 * n1 * n2;
  if (total == 0) return 0;
  long long blocks = (total + 255) / 256;
  if (blocks > 65536) blocks = 65536;
  k_gen_normal<<<(int)blocks, 256, 0, static_cast<cudaStream_t>(stream)>>>(a);
  return (int)cudaGetLastError();
}
