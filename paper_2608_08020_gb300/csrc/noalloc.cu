// Paged decode attention that allocates nothing.
//
// Some programs cannot allocate device memory at the point where they decode: a
// serving process that hands all of the GPU's memory to its own allocator when it
// starts and allows no allocation on the token path, or code that runs inside a
// framework whose device memory it does not own.  Such a caller already owns its KV
// pages, block tables, lengths, queries and output buffer, and passes exactly those.
// The working memory the call needs - the split-KV work plan and the partial results
// that the combine step merges - lives in one fixed array in this library's own
// device memory, so the call neither allocates nor asks the caller for a workspace.
//
// The array is a file-scope __device__ variable: every GPU that loads the library
// holds it (kNoAllocScratchBytes) until the process exits.  Host code cannot use the
// variable's name as a device address, so the address is looked up once per device
// with cudaGetSymbolAddress, with that device current, and passed to the kernels.
#include <mutex>

#include "internal.cuh"

namespace gb {
namespace {

constexpr size_t kNoAllocScratchBytes = 32ull << 20;  // 32 MiB
__device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocScratchBytes];

constexpr int kMaxDevices = 64;
std::mutex g_scratch_mu;
void* g_scratch_addr[kMaxDevices] = {};

// Device address of the scratch array on `device` (the current device); looked up on the
// first call for that device and remembered.
cudaError_t scratch_address(int device, void** out) {
  std::lock_guard<std::mutex> lock(g_scratch_mu);
  if (g_scratch_addr[device] == nullptr) {
    void* p = nullptr;
    const cudaError_t e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
    if (e != cudaSuccess) return e;
    g_scratch_addr[device] = p;
  }
  *out = g_scratch_addr[device];
  return cudaSuccess;
}

size_t round256(size_t x) { return (x + 255) & ~size_t(255); }

struct ScratchLayout {
  size_t ctl, active, plan, partials, total;
};

ScratchLayout scratch_layout(int beams, int Hkv, int W, int record_floats) {
  ScratchLayout s{};
  size_t o = 0;
  s.ctl = o;      o = round256(o + kCtlWords * sizeof(int));
  s.active = o;   o = round256(o + (size_t)beams * sizeof(int));
  s.plan = o;     o = round256(o + 3 * (size_t)(beams + 1) * sizeof(int));
  s.partials = o; o = round256(o + (size_t)(W + beams * Hkv) * record_floats * sizeof(float));
  s.total = o;
  return s;
}

// Work plan for caller-owned rows (one thread per row): every row with seq_len > 0 is
// read whole.  A row whose length is negative or longer than its table
// (max_pages_per_beam x page_size tokens) is not read at all: its output is zero and the
// call's status records GB_ERR_INVALID.  The status word, the one scratch value that must
// start at zero, is cleared first.
__global__ void __launch_bounds__(1024) k_noalloc_plan(PoolView v) {
  pdl_wait();
  pdl_launch_dependents();
  __shared__ int tmp[33];
  const int b = threadIdx.x;
  if (b == 0) v.ctl[kCtlStatus] = GB_OK;
  __syncthreads();
  const int L = b < v.max_beams ? v.seq_len[b] : 0;
  const bool bad = b < v.max_beams && (L < 0 || (long long)L > (long long)v.max_pages * v.P);
  if (bad) set_status(v.ctl, GB_ERR_INVALID);
  const bool act = L > 0 && !bad;
  const int n = act ? (L + kChunk - 1) / kChunk : 0;
  int total;
  const int off = block_exclusive_scan(n * v.Hkv, tmp, &total);
  if (b < v.max_beams) {
    v.active[b] = act ? 1 : 0;
    plan_off(v, 0)[b] = off;
    plan_n(v, 0)[b] = n;
    plan_start(v, 0)[b] = 0;
  }
  if (b == 0) {
    plan_off(v, 0)[v.max_beams] = total;
    v.ctl[kCtlStepOk] = 1;
  }
}

}  // namespace
}  // namespace gb

using namespace gb;

extern "C" gb_status gb_paged_decode_noalloc(const gb_paged_decode_args* a, gb_stream_t stream) {
  if (!a || !a->kv || !a->tables || !a->seq_len || !a->q || !a->out) return GB_ERR_INVALID;
  if (a->num_beams < 1 || a->num_beams > kMaxBeams || a->num_q_heads < 1 || a->num_kv_heads < 1 ||
      a->num_q_heads % a->num_kv_heads != 0 || a->max_pages_per_beam < 1 || a->num_pages < 1 ||
      a->num_pages > (int64_t)0x7fffffff)
    return GB_ERR_INVALID;
  if (!(a->page_size == 16 || a->page_size == 32 || a->page_size == 64)) return GB_ERR_INVALID;
  if (a->kv_dtype != GB_F32 && a->kv_dtype != GB_BF16) return GB_ERR_INVALID;
  const int G = a->num_q_heads / a->num_kv_heads;
  if (!decode_supported(a->kv_dtype, a->head_dim, G)) return GB_ERR_UNSUPPORTED;
  if (((uintptr_t)a->kv & 15) || ((uintptr_t)a->q & 15)) return GB_ERR_INVALID;
  // The work plan counts 16-token chunks per (row, KV head) in 32-bit integers.
  const long long max_chunks = ((long long)a->max_pages_per_beam * a->page_size + kChunk - 1) / kChunk;
  if ((long long)a->num_beams * max_chunks * a->num_kv_heads >= (1ll << 31)) return GB_ERR_INVALID;

  int device = 0, sms = 0;
  if (cudaGetDevice(&device) != cudaSuccess || device < 0 || device >= kMaxDevices) return GB_ERR_CUDA;
  if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, device) != cudaSuccess) return GB_ERR_CUDA;
  const int W = sms * kDecodeWarps < kMaxDecodeWarps ? sms * kDecodeWarps : kMaxDecodeWarps;
  const int record_floats = G * (a->head_dim + 2);
  const ScratchLayout L = scratch_layout(a->num_beams, a->num_kv_heads, W, record_floats);
  if (L.total > kNoAllocScratchBytes) return GB_ERR_TOO_LARGE;

  void* base = nullptr;
  if (scratch_address(device, &base) != cudaSuccess) return GB_ERR_CUDA;
  char* sc = static_cast<char*>(base);

  PoolView v{};
  v.layers = 1;
  v.Hq = a->num_q_heads;
  v.Hkv = a->num_kv_heads;
  v.D = a->head_dim;
  v.P = a->page_size;
  v.G = G;
  v.dtype = a->kv_dtype;
  v.esize = a->kv_dtype == GB_BF16 ? 2 : 4;
  v.max_beams = a->num_beams;
  v.max_pages = a->max_pages_per_beam;
  v.num_pages = a->num_pages;
  v.kv = static_cast<char*>(const_cast<void*>(a->kv));
  v.page_elems = 2LL * v.Hkv * v.P * v.D;
  v.tables = const_cast<int*>(a->tables);
  v.seq_len = const_cast<int*>(a->seq_len);
  v.ctl = reinterpret_cast<int*>(sc + L.ctl);
  v.active = reinterpret_cast<int*>(sc + L.active);
  v.plan = reinterpret_cast<int*>(sc + L.plan);
  v.partials = reinterpret_cast<float*>(sc + L.partials);
  v.record_floats = record_floats;

  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  k_noalloc_plan<<<1, 1024, 0, s>>>(v);
  if (cudaGetLastError() != cudaSuccess) return GB_ERR_CUDA;
  if (launch_decode_view(v, W, 0, a->q, a->scale, a->out, s) != cudaSuccess) return GB_ERR_CUDA;
  return GB_OK;
}

extern "C" gb_status gb_paged_decode_noalloc_status(int* device_status, gb_stream_t stream) {
  if (!device_status) return GB_ERR_INVALID;
  int device = 0;
  if (cudaGetDevice(&device) != cudaSuccess || device < 0 || device >= kMaxDevices) return GB_ERR_CUDA;
  void* base = nullptr;
  if (scratch_address(device, &base) != cudaSuccess) return GB_ERR_CUDA;
  // The status word is the first word of the scratch array (ScratchLayout::ctl = 0).
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  int v = GB_OK;
  if (cudaMemcpyAsync(&v, static_cast<const int*>(base) + kCtlStatus, sizeof(int), cudaMemcpyDeviceToHost, s) !=
          cudaSuccess ||
      cudaStreamSynchronize(s) != cudaSuccess)
    return GB_ERR_CUDA;
  *device_status = v;
  return GB_OK;
}
