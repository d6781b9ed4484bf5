// Paged KV pool: creation, seeding, per-step page reservation, KV append and
// release.  Pages are refcounted; a branched child shares its parent's pages
// (Section 3.1, after Eq. 3: the child inherits the parent's KV through prefix
// caching) and pruning frees only pages nobody else references.
//
// Allocation rule: the lowest free page id, slots served in ascending order,
// token by token.  Planners run as a single CTA with one thread per slot so
// the order is exactly that sequential rule.
#include <algorithm>
#include <cstring>
#include <mutex>
#include <set>
#include <tuple>
#include <vector>

#include "internal.cuh"

namespace gb {

static size_t align256(size_t x) { return (x + 255) & ~size_t(255); }

MetaLayout meta_layout(const gb_pool_config& c) {
  MetaLayout m{};
  const size_t B = (size_t)c.max_beams;
  const int G = c.num_q_heads / c.num_kv_heads;
  size_t o = 0;
  auto take = [&](size_t bytes) { size_t at = o; o = align256(o + bytes); return at; };
  m.ctl = take(kCtlWords * sizeof(int));
  m.tables = take(B * c.max_pages_per_beam * sizeof(int));
  m.seq_len = take(B * sizeof(int));
  m.active = take(B * sizeof(int));
  m.gen = take(B * sizeof(int));
  m.nsteps = take(B * sizeof(int));
  m.mean = take(B * sizeof(float));
  m.lineage = take(B * sizeof(unsigned));
  m.refcnt = take((size_t)c.num_pages * sizeof(int));
  m.words = (int)((c.num_pages + 31) / 32);
  m.free_bits = take((size_t)m.words * sizeof(unsigned));
  m.plan = take(2 * 3 * (B + 1) * sizeof(int));
  m.cow = take(kMaxCowJobs * 3 * sizeof(int));
  m.record_floats = G * (c.head_dim + 2);
  m.partial_records = kMaxDecodeWarps + (int)B * c.num_kv_heads;  // record index: warp + b * Hkv + h
  m.partials = take((size_t)m.partial_records * m.record_floats * sizeof(float));
  const size_t BD = B * kMaxSegDepth;
  m.seg_cover = take(B * sizeof(int));
  m.seg_nseg = take(B * sizeof(int));
  m.seg_owner = take((size_t)c.num_pages * sizeof(unsigned long long));
  m.seg_i0 = take(BD * sizeof(int));
  m.seg_len = take(BD * sizeof(int));
  m.seg_rep = take(BD * sizeof(int));
  m.seg_g = take(BD * sizeof(int));
  m.seg_mem_off = take(BD * sizeof(int));
  m.seg_fill = take(BD * sizeof(int));
  m.seg_members = take(BD * sizeof(int));
  m.seg_tile_seg = take(B * kMaxSegRecords * sizeof(int));  // work entries <= records
  m.seg_tile_t = take(B * kMaxSegRecords * sizeof(int));
  m.grec = take(B * kMaxSegRecords * c.num_kv_heads * m.record_floats * sizeof(float));
  m.seg_bid = take(BD * sizeof(int));
  m.seg_rec_off = take(BD * sizeof(int));
  m.seg_nrec = take(B * sizeof(int));
  m.seg_splits = take(BD * sizeof(int));
  m.seg_tile_split = take(B * kMaxSegRecords * sizeof(int));
  m.seg_hist = take(2 * 256 * sizeof(int));
  m.pair_cnt = take(B * c.num_kv_heads * sizeof(int));
  m.stats = take((size_t)kStatsRing * kStatsWords * sizeof(int));
  m.mlp_scratch = take((size_t)kMlpScratchFloats * sizeof(float));
  m.total = o;
  return m;
}

bool decode_supported(int dtype, int D, int G) {
  if (!(G == 2 || G == 4 || G == 8)) return false;
  if (dtype == GB_BF16) return D == 128;
  if (dtype == GB_F32) return D == 64;
  return false;
}

gb_status fail(gb_pool* pool, gb_status code, const char* what) {
  if (pool) pool->last_error = what;
  return code;
}

cudaError_t set_max_dynamic_smem(const void* kernel, int bytes) {
  static std::mutex mu;
  static std::set<std::tuple<const void*, int, int>> done;  // (kernel, device, bytes) already set
  int device = 0;
  cudaError_t e = cudaGetDevice(&device);
  if (e != cudaSuccess) return e;
  std::lock_guard<std::mutex> lock(mu);
  if (done.count(std::make_tuple(kernel, device, bytes))) return cudaSuccess;
  e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
  if (e == cudaSuccess) done.insert(std::make_tuple(kernel, device, bytes));
  return e;
}

gb_status check_launch(gb_pool* pool, const char* what) {
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) {
    if (pool) pool->last_error = std::string(what) + ": " + cudaGetErrorString(e);
    return GB_ERR_CUDA;
  }
  return GB_OK;
}

// ---------------------------------------------------------------------------
// Device helpers
// ---------------------------------------------------------------------------

// Block-wide search for the `need` lowest free pages, starting at the cursor
// word.  Writes them ascending into out[0..need).  Returns the number found
// (uniform).  Does not modify the bitmap.
__device__ int find_lowest_free(const PoolView& v, int need, int* out, int* tmp) {
  int found = 0;
  int w0 = v.ctl[kCtlCursor];
  if (w0 < 0) w0 = 0;
  while (found < need && w0 < v.words) {
    const int w = w0 + threadIdx.x;
    unsigned bits = w < v.words ? v.free_bits[w] : 0u;
    if (w == v.words - 1 && (v.num_pages & 31)) bits &= (1u << (v.num_pages & 31)) - 1u;
    int total;
    int r = found + block_exclusive_scan(__popc(bits), tmp, &total);
    while (bits && r < need) {
      const int bit = __ffs(bits) - 1;
      bits &= bits - 1u;
      out[r++] = w * 32 + bit;
    }
    found += total;
    w0 += blockDim.x;
  }
  __syncthreads();
  return found < need ? found : need;
}

// Take pages out[0..n) from the free set (bitmap, count, cursor).
__device__ void take_pages(const PoolView& v, const int* pages, int n) {
  for (int r = threadIdx.x; r < n; r += blockDim.x) {
    const int p = pages[r];
    atomicAnd(&v.free_bits[p >> 5], ~(1u << (p & 31)));
  }
  if (threadIdx.x == 0 && n > 0) {
    v.ctl[kCtlFree] -= n;
    v.ctl[kCtlCursor] = pages[n - 1] >> 5;
  }
  __syncthreads();
}

// ---------------------------------------------------------------------------
// Kernels
// ---------------------------------------------------------------------------

__global__ void k_init(PoolView v) {
  pdl_wait();
  pdl_launch_dependents();
  const long long tid = blockIdx.x * (long long)blockDim.x + threadIdx.x;
  const long long stride = (long long)gridDim.x * blockDim.x;
  for (long long w = tid; w < v.words; w += stride) {
    unsigned bits = 0xffffffffu;
    if (w == v.words - 1 && (v.num_pages & 31)) bits = (1u << (v.num_pages & 31)) - 1u;
    v.free_bits[w] = bits;
  }
  for (long long i = tid; i < (long long)v.max_beams * v.max_pages; i += stride) v.tables[i] = -1;
  if (tid == 0) {
    for (int i = 0; i < kCtlWords; ++i) v.ctl[i] = 0;
    v.ctl[kCtlNextLineage] = 1;
    v.ctl[kCtlFree] = (int)v.num_pages;
  }
}

// Reserve the prompt's pages for n root beams (one CTA).
__global__ void __launch_bounds__(1024) k_seed_alloc(PoolView v, int n_beams, int prompt_len) {
  pdl_wait();
  pdl_launch_dependents();
  __shared__ int tmp[33];
  __shared__ int s_pages[2048];
  const int npg = (prompt_len + v.P - 1) / v.P;
  if (npg > v.max_pages || npg > 2048 || npg > v.ctl[kCtlFree]) {
    if (threadIdx.x == 0) { set_status(v.ctl, GB_ERR_OOM); v.ctl[kCtlStepOk] = 0; }
    return;
  }
  const int got = find_lowest_free(v, npg, s_pages, tmp);
  if (got < npg) {
    if (threadIdx.x == 0) set_status(v.ctl, GB_ERR_OOM);
    return;
  }
  take_pages(v, s_pages, npg);
  for (int i = threadIdx.x; i < npg; i += blockDim.x) v.refcnt[s_pages[i]] = n_beams;
  for (int i = threadIdx.x; i < n_beams * npg; i += blockDim.x)
    v.tables[(size_t)(i / npg) * v.max_pages + (i % npg)] = s_pages[i % npg];
  const int lin0 = v.ctl[kCtlNextLineage];
  __syncthreads();
  for (int b = threadIdx.x; b < n_beams; b += blockDim.x) {
    v.seq_len[b] = prompt_len;
    v.active[b] = 1;
    v.gen[b] = 0;
    v.nsteps[b] = 0;
    v.mean[b] = 0.f;
    v.lineage[b] = (unsigned)(lin0 + b);
  }
  if (threadIdx.x == 0) {
    v.ctl[kCtlNextLineage] = lin0 + n_beams;
    v.ctl[kCtlTailShared] = 1;  // the prompt's last page may be partial
  }
}

// Copy the prompt's K/V ([layer][T][Hkv][D]) into the pages listed in slot 0's table.
__global__ void k_seed_write(PoolView v, int prompt_len, const char* kp, const char* vp) {
  pdl_wait();
  pdl_launch_dependents();
  const int vec_per_row = v.D * v.esize / 16;
  const long long rows = (long long)v.layers * prompt_len * v.Hkv;
  const long long total = rows * vec_per_row * 2;
  for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < total;
       i += (long long)gridDim.x * blockDim.x) {
    const int kv = (int)(i / (rows * vec_per_row));
    long long r = i % (rows * vec_per_row);
    const int vec = (int)(r % vec_per_row);
    r /= vec_per_row;
    const int head = (int)(r % v.Hkv);
    r /= v.Hkv;
    const int t = (int)(r % prompt_len);
    const int layer = (int)(r / prompt_len);
    const int page = v.tables[t / v.P];
    if (page < 0 || page >= v.num_pages) continue;
    const char* src = (kv ? vp : kp) + ((((long long)layer * prompt_len + t) * v.Hkv + head) * v.D) * v.esize;
    char* dst = v.kv + kv_elem_offset(v, layer, page, kv, head, t % v.P) * v.esize;
    reinterpret_cast<uint4*>(dst)[vec] = reinterpret_cast<const uint4*>(src)[vec];
  }
}

// Open a step of n_tokens tokens for every active slot (one CTA, thread = slot):
// reserve pages in the sequential order (token by token, slots ascending),
// copy still-shared partial tail pages, advance lengths, build decode plans.
// All or nothing: if the pool cannot supply every page the step is a no-op.
__global__ void __launch_bounds__(1024) k_step_begin(PoolView v, int n_tokens, const int* seg_cover) {
  pdl_wait();
  pdl_launch_dependents();
  __shared__ int tmp[33];
  __shared__ int s_alloc[kMaxBeams];
  __shared__ int s_tail[kMaxBeams];
  __shared__ int s_ncow, s_nact;
  __shared__ int s_tok[2];
  __shared__ int s_ctl[8];  // free pages, steps, and the segment totals of the step record
  const int b = threadIdx.x;
  // Every load that depends on nothing else goes out first, together.
  const bool act = b < v.max_beams && v.active[b] != 0;
  const int L = act ? v.seq_len[b] : 0;
  const int cover = (seg_cover != nullptr && b < v.max_beams) ? seg_cover[b] : 0;
  if (b == 0) {
    s_ncow = 0;
    s_ctl[0] = v.ctl[kCtlFree];
    s_ctl[1] = v.ctl[kCtlSteps];
    s_ctl[2] = v.ctl[kCtlSegRowTok];
    s_ctl[3] = v.ctl[kCtlSegTileTok];
    s_ctl[4] = v.ctl[kCtlSegCount];
    s_ctl[5] = v.ctl[kCtlSegTiles];
    s_ctl[6] = v.ctl[kCtlSegTok];
    s_ctl[7] = v.ctl[kCtlTailShared];
  }

  // Copy-on-write decision for a still-shared partial tail page: holders
  // decide in slot order against the current refcount, so the i-th holder
  // (1-based) copies iff i < refcnt.  Only after a seed or a fork can a partial tail page be
  // shared; the first step after one resolves them all.
  __syncthreads();
  const bool tails_shared = s_ctl[7] != 0;
  int tail = -1;
  if (tails_shared && act && (L % v.P) != 0) tail = v.tables[(size_t)b * v.max_pages + L / v.P];
  if (b < kMaxBeams) s_tail[b] = tail;
  __syncthreads();
  bool cow = false;
  if (tail >= 0) {
    const int R = v.refcnt[tail];
    if (R > 1) {
      int i = 1;
      for (int o = 0; o < b; ++o) i += (s_tail[o] == tail);
      cow = i < R;
    }
  }
  // Pages this slot needs over the whole step, and the table capacity check.
  int need_total = 0;
  bool too_long = false;
  if (act) {
    const int first_new = (L + v.P - 1) / v.P;        // first page index that needs a fresh page
    const int last_idx = (L + n_tokens - 1) / v.P;    // page index of the last new token
    need_total = (last_idx >= first_new ? last_idx - first_new + 1 : 0) + (cow ? 1 : 0);
    too_long = last_idx >= v.max_pages;
  }
  int total_need, nact;
  block_exclusive_scan(need_total, tmp, &total_need);
  block_exclusive_scan(act ? 1 : 0, tmp, &nact);
  if (b == 0) s_nact = nact;
  const bool any_too_long = __syncthreads_or(too_long);
  if (any_too_long || total_need > s_ctl[0]) {
    if (b == 0) v.ctl[kCtlCowJobs] = 0;
    if (b == 0) { set_status(v.ctl, GB_ERR_OOM); v.ctl[kCtlStepOk] = 0; }
    return;
  }

  for (int k = 0; k < n_tokens; ++k) {
    const int pos = L + k;
    const bool need_new = act && (pos % v.P) == 0;
    const bool need = need_new || (k == 0 && cow);
    if (!__syncthreads_or(need)) continue;
    int n_need;
    const int rank = block_exclusive_scan(need ? 1 : 0, tmp, &n_need);
    const int got = find_lowest_free(v, n_need, s_alloc, tmp);
    if (got < n_need) {  // cannot happen after the count check; keep the pool consistent
      if (b == 0) { set_status(v.ctl, GB_ERR_OOM); v.ctl[kCtlStepOk] = 0; }
      return;
    }
    take_pages(v, s_alloc, n_need);
    if (need) {
      const int page = s_alloc[rank];
      v.refcnt[page] = 1;
      v.tables[(size_t)b * v.max_pages + pos / v.P] = page;
      if (!need_new) {  // copy-on-write of the shared tail page
        atomicSub(&v.refcnt[tail], 1);
        const int j = atomicAdd(&s_ncow, 1);
        if (j < kMaxCowJobs) {
          v.cow[3 * j] = tail;
          v.cow[3 * j + 1] = page;
          v.cow[3 * j + 2] = L % v.P;
        }
      }
    }
    __syncthreads();
  }
  // The rows [0, L % P) of each copied page are copied layer by layer by the append kernel.
  if (b == 0) v.ctl[kCtlCowJobs] = min(s_ncow, kMaxCowJobs);

  const int Lnew = act ? L + n_tokens : 0;
  if (act) {
    v.seq_len[b] = Lnew;
    v.gen[b] += n_tokens;
  }
  // Decode plans: mode 0 reads every token per beam; mode 1 skips the prefix
  // covered by grouped shared-prefix segments.
  for (int mode = 0; mode < 2; ++mode) {
    int start = 0;
    if (mode == 1 && act) start = cover * v.P;
    if (start > Lnew) start = Lnew;
    const int n = act ? (Lnew - start + kChunk - 1) / kChunk : 0;
    int total;
    const int off = block_exclusive_scan(n * v.Hkv, tmp, &total);
    if (b < v.max_beams) {
      plan_off(v, mode)[b] = off;
      plan_n(v, mode)[b] = n;
      plan_start(v, mode)[b] = start;
    }
    if (b == 0) plan_off(v, mode)[v.max_beams] = total;
    int tok_total;
    block_exclusive_scan(act ? Lnew - start : 0, tmp, &tok_total);
    if (b == 0) s_tok[mode] = tok_total;
  }
  if (b == 0) {
    // Work of this step: tokens each path reads per KV head, and the segment work of the
    // grouped path (valid until the next rebuild).
    const int step = s_ctl[1];
    int* e = v.stats + (size_t)(step % kStatsRing) * kStatsWords;
    e[0] = s_tok[0];
    e[1] = s_tok[1];
    e[2] = v.grouped ? s_ctl[2] : 0;
    e[3] = v.grouped ? s_ctl[3] : 0;
    e[4] = v.grouped ? s_ctl[4] : 0;
    e[5] = v.grouped ? s_ctl[5] : 0;
    e[6] = n_tokens;
    e[7] = step;
    e[8] = v.grouped ? s_ctl[6] : 0;
    e[9] = s_nact;
    v.ctl[kCtlSteps] = step + 1;
  }
  if (b == 0) {
    if (tails_shared) v.ctl[kCtlTailShared] = 0;
    v.ctl[kCtlStepOk] = 1;
  }
}

// Write n_tokens new K/V rows per active slot for one layer at positions
// [seq_len - n_tokens, seq_len).  kin/vin: [n_tokens][max_beams][Hkv][D].
__global__ void k_append(PoolView v, int layer, int n_tokens, const char* kin, const char* vin) {
  pdl_wait();
  pdl_launch_dependents();
  // The counters of the attention launch that follows (combine.cuh, the grouped role's
  // work queue): the previous attention launch has completed (pdl_wait).
  if (blockIdx.x == 0 && blockIdx.y == 0) {
    for (int i = threadIdx.x; i < v.max_beams * v.Hkv; i += blockDim.x) v.pair_cnt[i] = 0;
    if (threadIdx.x == 0) {
      v.ctl[kCtlGrpNext] = 0;
      v.ctl[kCtlGrpDone] = 0;
      v.ctl[kCtlPairNext] = 0;
    }
  }
  if (v.ctl[kCtlStepOk] == 0) return;
  const int vec_per_row = v.D * v.esize / 16;
  // Copy-on-write of still-shared partial tail pages, this layer's rows [0, rows).
  // Rows differ from every row written below, so both loops run concurrently.
  const int ncow = v.ctl[kCtlCowJobs];
  const long long per_job = 2LL * v.Hkv * v.P * vec_per_row;
  const long long nthreads = (long long)gridDim.x * gridDim.y * blockDim.x;
  for (long long i = ((long long)blockIdx.y * gridDim.x + blockIdx.x) * blockDim.x + threadIdx.x; i < per_job * ncow;
       i += nthreads) {
    const int j = (int)(i / per_job);
    long long r = i % per_job;
    const int vec = (int)(r % vec_per_row); r /= vec_per_row;
    const int row = (int)(r % v.P); r /= v.P;
    if (row >= v.cow[3 * j + 2]) continue;
    const int head = (int)(r % v.Hkv);
    const int kv = (int)(r / v.Hkv);
    const uint4* src = reinterpret_cast<const uint4*>(v.kv + kv_elem_offset(v, layer, v.cow[3 * j], kv, head, row) * v.esize);
    uint4* dst = reinterpret_cast<uint4*>(v.kv + kv_elem_offset(v, layer, v.cow[3 * j + 1], kv, head, row) * v.esize);
    dst[vec] = src[vec];
  }
  // New rows: blockIdx.y walks (K|V, token), x covers (slot, head, 16-byte vector) with
  // 32-bit index arithmetic (a row is 256 bytes, 16 vectors, for every supported shape).
  const int per_tok = v.max_beams * v.Hkv * vec_per_row;
  for (int y = blockIdx.y; y < 2 * n_tokens; y += gridDim.y) {
    const int kv = y >= n_tokens ? 1 : 0;
    const int k = y - kv * n_tokens;
    for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < per_tok; i += gridDim.x * blockDim.x) {
      const int vec = i & 15;
      const int r = i >> 4;
      const int b = r / v.Hkv, head = r - b * v.Hkv;
      if (!v.active[b]) continue;
      const int pos = v.seq_len[b] - n_tokens + k;
      if (pos < 0) continue;
      const int page = v.tables[(size_t)b * v.max_pages + pos / v.P];
      if (page < 0 || page >= v.num_pages) { set_status(v.ctl, GB_ERR_INVALID); continue; }
      const char* src = (kv ? vin : kin) + ((((long long)k * v.max_beams + b) * v.Hkv + head) * v.D) * v.esize;
      char* dst = v.kv + kv_elem_offset(v, layer, page, kv, head, pos % v.P) * v.esize;
      reinterpret_cast<uint4*>(dst)[vec] = reinterpret_cast<const uint4*>(src)[vec];
    }
  }
}

// Release listed slots in order (one CTA).
__global__ void __launch_bounds__(1024) k_release(PoolView v, const int* slots, int n) {
  pdl_wait();
  pdl_launch_dependents();
  for (int i = 0; i < n; ++i) {
    const int s = slots[i];
    if (s < 0 || s >= v.max_beams) {
      if (threadIdx.x == 0) set_status(v.ctl, GB_ERR_INVALID);
      continue;
    }
    if (!v.active[s]) {
      if (threadIdx.x == 0) set_status(v.ctl, GB_ERR_STATE);
      __syncthreads();
      continue;
    }
    const int npg = (v.seq_len[s] + v.P - 1) / v.P;
    for (int j = threadIdx.x; j < npg; j += blockDim.x) {
      const int p = v.tables[(size_t)s * v.max_pages + j];
      if (p >= 0 && p < v.num_pages) unref_page(v, p);
    }
    __syncthreads();
    if (threadIdx.x == 0) {
      v.active[s] = 0;
      v.seq_len[s] = 0;
      v.gen[s] = 0;
    }
    __threadfence_block();
    __syncthreads();
  }
}

__global__ void k_clear_status(PoolView v) {
  pdl_wait();
  pdl_launch_dependents(); v.ctl[kCtlStatus] = GB_OK; }

}  // namespace gb

using namespace gb;

// ---------------------------------------------------------------------------
// C ABI
// ---------------------------------------------------------------------------

static gb_status validate(const gb_pool_config* c) {
  if (!c) return GB_ERR_INVALID;
  if (c->num_layers < 1 || c->num_q_heads < 1 || c->num_kv_heads < 1 ||
      c->num_q_heads % c->num_kv_heads != 0 || c->head_dim < 1 || c->num_pages < 1 ||
      c->num_pages > (int64_t)0x7fffffff || c->max_beams < 1 || c->max_beams > kMaxBeams ||
      c->max_pages_per_beam < 1 || c->group_min_beams < 0)
    return GB_ERR_INVALID;
  if (!(c->page_size == 16 || c->page_size == 32 || c->page_size == 64)) return GB_ERR_INVALID;
  if (c->kv_dtype != GB_F32 && c->kv_dtype != GB_BF16) return GB_ERR_INVALID;
  if (!decode_supported(c->kv_dtype, c->head_dim, c->num_q_heads / c->num_kv_heads))
    return GB_ERR_UNSUPPORTED;
  return GB_OK;
}

static size_t kv_bytes_of(const gb_pool_config* c) {
  const size_t es = c->kv_dtype == GB_BF16 ? 2 : 4;
  return (size_t)c->num_layers * (size_t)c->num_pages * 2 * c->num_kv_heads * c->page_size *
         c->head_dim * es;
}

extern "C" gb_status gb_pool_workspace_bytes(const gb_pool_config* cfg, size_t* kv_bytes,
                                             size_t* meta_bytes) {
  gb_status st = validate(cfg);
  if (st != GB_OK) return st;
  if (kv_bytes) *kv_bytes = kv_bytes_of(cfg);
  if (meta_bytes) *meta_bytes = meta_layout(*cfg).total;
  return GB_OK;
}

extern "C" gb_status gb_pool_init(const gb_pool_config* cfg, void* kv_dev, void* meta_dev,
                                  gb_stream_t stream, gb_pool** out) {
  if (!out) return GB_ERR_INVALID;
  *out = nullptr;
  gb_status st = validate(cfg);
  if (st != GB_OK) return st;
  if (!kv_dev || !meta_dev || ((uintptr_t)kv_dev & 255) || ((uintptr_t)meta_dev & 255))
    return GB_ERR_INVALID;
  gb_pool* p = new gb_pool();
  p->cfg = *cfg;
  p->layout = meta_layout(*cfg);
  if (cudaGetDevice(&p->device) != cudaSuccess ||
      cudaDeviceGetAttribute(&p->num_sms, cudaDevAttrMultiProcessorCount, p->device) != cudaSuccess) {
    delete p;
    return GB_ERR_CUDA;
  }
  p->decode_warps = std::min(kMaxDecodeWarps, p->num_sms * kDecodeCtasPerSm * kDecodeWarps);
  p->next_layer = 0;
  p->step_tokens = 0;
  p->seeded = false;
  p->group_min = cfg->group_min_beams > 0 ? cfg->group_min_beams : 2;
  PoolView& v = p->view;
  v.layers = cfg->num_layers;
  v.Hq = cfg->num_q_heads;
  v.Hkv = cfg->num_kv_heads;
  v.D = cfg->head_dim;
  v.P = cfg->page_size;
  v.G = v.Hq / v.Hkv;
  v.dtype = cfg->kv_dtype;
  v.esize = cfg->kv_dtype == GB_BF16 ? 2 : 4;
  v.max_beams = cfg->max_beams;
  v.max_pages = cfg->max_pages_per_beam;
  v.words = p->layout.words;
  v.num_pages = cfg->num_pages;
  v.kv = static_cast<char*>(kv_dev);
  v.page_elems = 2LL * v.Hkv * v.P * v.D;
  char* m = static_cast<char*>(meta_dev);
  const MetaLayout& L = p->layout;
  v.ctl = reinterpret_cast<int*>(m + L.ctl);
  v.tables = reinterpret_cast<int*>(m + L.tables);
  v.seq_len = reinterpret_cast<int*>(m + L.seq_len);
  v.active = reinterpret_cast<int*>(m + L.active);
  v.gen = reinterpret_cast<int*>(m + L.gen);
  v.nsteps = reinterpret_cast<int*>(m + L.nsteps);
  v.mean = reinterpret_cast<float*>(m + L.mean);
  v.lineage = reinterpret_cast<unsigned*>(m + L.lineage);
  v.refcnt = reinterpret_cast<int*>(m + L.refcnt);
  v.free_bits = reinterpret_cast<unsigned*>(m + L.free_bits);
  v.plan = reinterpret_cast<int*>(m + L.plan);
  v.cow = reinterpret_cast<int*>(m + L.cow);
  v.partials = reinterpret_cast<float*>(m + L.partials);
  v.record_floats = L.record_floats;
  v.seg_cover = reinterpret_cast<int*>(m + L.seg_cover);
  v.seg_nseg = reinterpret_cast<int*>(m + L.seg_nseg);
  v.seg_owner = reinterpret_cast<unsigned long long*>(m + L.seg_owner);
  v.seg_i0 = reinterpret_cast<int*>(m + L.seg_i0);
  v.seg_len = reinterpret_cast<int*>(m + L.seg_len);
  v.seg_rep = reinterpret_cast<int*>(m + L.seg_rep);
  v.seg_g = reinterpret_cast<int*>(m + L.seg_g);
  v.seg_mem_off = reinterpret_cast<int*>(m + L.seg_mem_off);
  v.seg_fill = reinterpret_cast<int*>(m + L.seg_fill);
  v.seg_members = reinterpret_cast<int*>(m + L.seg_members);
  v.seg_tile_seg = reinterpret_cast<int*>(m + L.seg_tile_seg);
  v.seg_tile_t = reinterpret_cast<int*>(m + L.seg_tile_t);
  v.grec = reinterpret_cast<float*>(m + L.grec);
  v.seg_bid = reinterpret_cast<int*>(m + L.seg_bid);
  v.seg_rec_off = reinterpret_cast<int*>(m + L.seg_rec_off);
  v.seg_nrec = reinterpret_cast<int*>(m + L.seg_nrec);
  v.seg_splits = reinterpret_cast<int*>(m + L.seg_splits);
  v.seg_tile_split = reinterpret_cast<int*>(m + L.seg_tile_split);
  v.seg_hist = reinterpret_cast<int*>(m + L.seg_hist);
  v.pair_cnt = reinterpret_cast<int*>(m + L.pair_cnt);
  v.num_sms = p->num_sms;
  v.stats = reinterpret_cast<int*>(m + L.stats);
  v.mlp_scratch = reinterpret_cast<float*>(m + L.mlp_scratch);
  v.group_min = p->group_min;
  // The grouped tensor-core path needs bf16 K/V with D = 128 (kind::f16 MMAs, 128-byte rows)
  // and pages of 8 to 64 tokens that tile a 64-token K/V tile exactly.
  v.grouped = (cfg->kv_dtype == GB_BF16 && cfg->head_dim == 128 && cfg->page_size % 8 == 0 &&
               64 % cfg->page_size == 0)
                  ? 1
                  : 0;
  make_kv_tensor_maps(p);
  // The grouped path runs as a role of the attention kernel beside the per-beam role, so it
  // needs both tensor maps.
  if (v.grouped && !(p->have_tmap && p->have_dtmap && p->num_sms * kMmaWarps <= kMaxDecodeWarps)) v.grouped = 0;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (cudaMemsetAsync(m, 0, L.partials, s) != cudaSuccess ||
      cudaMemsetAsync(m + L.seg_cover, 0, L.seg_owner - L.seg_cover, s) != cudaSuccess ||
      cudaMemsetAsync(m + L.seg_owner, 0, (size_t)cfg->num_pages * sizeof(unsigned long long), s) != cudaSuccess) {
    delete p;
    return GB_ERR_CUDA;
  }
  p->launches += 1;
  k_init<<<std::max(1, std::min(p->num_sms * 4, (int)((v.max_beams * (long long)v.max_pages + 255) / 256))), 256, 0, s>>>(v);
  st = check_launch(p, "init");
  if (st != GB_OK) {
    delete p;
    return st;
  }
  *out = p;
  return GB_OK;
}

extern "C" gb_status gb_pool_destroy(gb_pool* pool) {
  delete pool;
  return GB_OK;
}

extern "C" const char* gb_last_error(gb_pool* pool) {
  return pool ? pool->last_error.c_str() : "";
}

extern "C" gb_status gb_pool_seed(gb_pool* pool, int n_beams, int prompt_len, const void* k_prompt_dev,
                                  const void* v_prompt_dev, gb_stream_t stream) {
  if (!pool) return GB_ERR_INVALID;
  if (pool->seeded) return fail(pool, GB_ERR_STATE, "seed: pool already seeded");
  if (n_beams < 1 || n_beams > pool->cfg.max_beams || prompt_len < 1 || !k_prompt_dev || !v_prompt_dev)
    return fail(pool, GB_ERR_INVALID, "seed: bad arguments");
  if ((prompt_len + pool->cfg.page_size - 1) / pool->cfg.page_size > 2048)
    return fail(pool, GB_ERR_UNSUPPORTED, "seed: prompt longer than 2048 pages");
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  k_seed_alloc<<<1, 1024, 0, s>>>(pool->view, n_beams, prompt_len);
  pool->launches += 2;
  gb_status st = check_launch(pool, "seed_alloc");
  if (st != GB_OK) return st;
  const long long vecs = 2LL * pool->cfg.num_layers * prompt_len * pool->cfg.num_kv_heads *
                         (pool->view.D * pool->view.esize / 16);
  const int grid = (int)std::min<long long>((vecs + 255) / 256, pool->num_sms * 8LL);
  k_seed_write<<<std::max(grid, 1), 256, 0, s>>>(pool->view, prompt_len,
                                                 static_cast<const char*>(k_prompt_dev),
                                                 static_cast<const char*>(v_prompt_dev));
  st = check_launch(pool, "seed_write");
  if (st != GB_OK) return st;
  pool->seeded = true;
  if (rebuild_segments(pool, s) != cudaSuccess) return check_launch(pool, "segments");
  return GB_OK;
}

// Shared by gb_decode_attention and gb_append_kv: open the step at layer 0
// and write the new rows of `layer`.
static gb_status append_layer(gb_pool* pool, int layer, int n_tokens, const void* k, const void* v,
                              cudaStream_t s) {
  if (!pool->seeded) return fail(pool, GB_ERR_STATE, "pool not seeded");
  if (layer < 0 || layer >= pool->cfg.num_layers || n_tokens < 1 || !k || !v)
    return fail(pool, GB_ERR_INVALID, "append: bad arguments");
  if (layer != pool->next_layer) return fail(pool, GB_ERR_STATE, "layers of a step must be called in order");
  if (layer == 0) {
    prof_begin(pool, GB_PROF_PLAN, s);
    // One thread per slot (rounded up to a warp): the planner's block scans span only the pool's slots.
    launch_pdl(k_step_begin, 1, std::max(32, (pool->cfg.max_beams + 31) / 32 * 32), 0, s, pool->view, n_tokens,
               pool->view.grouped ? pool->view.seg_cover : nullptr);
    prof_end(pool, GB_PROF_PLAN, s);
    pool->launches += 1;
    gb_status st = check_launch(pool, "step_begin");
    if (st != GB_OK) return st;
    pool->step_tokens = n_tokens;
  } else if (n_tokens != pool->step_tokens) {
    return fail(pool, GB_ERR_STATE, "token count differs from the one layer 0 reserved");
  }
  const int per_tok = pool->cfg.max_beams * pool->cfg.num_kv_heads * (pool->view.D * pool->view.esize / 16);
  const dim3 grid(std::max(1, std::min((per_tok + 255) / 256, pool->num_sms * 8)), std::min(2 * n_tokens, 65535));
  prof_begin(pool, GB_PROF_APPEND, s);
  launch_pdl(k_append, grid, 256, 0, s, pool->view, layer, n_tokens, static_cast<const char*>(k),
             static_cast<const char*>(v));
  prof_end(pool, GB_PROF_APPEND, s);
  pool->launches += 1;
  gb_status st = check_launch(pool, "append");
  if (st != GB_OK) return st;
  pool->next_layer = (layer + 1) % pool->cfg.num_layers;
  return GB_OK;
}

extern "C" gb_status gb_append_kv(gb_pool* pool, int layer, int n_tokens, const void* k_dev,
                                  const void* v_dev, gb_stream_t stream) {
  if (!pool) return GB_ERR_INVALID;
  return append_layer(pool, layer, n_tokens, k_dev, v_dev, reinterpret_cast<cudaStream_t>(stream));
}

extern "C" gb_status gb_decode_attention(gb_pool* pool, int layer, const void* q_dev,
                                         const void* k_new_dev, const void* v_new_dev, float scale,
                                         float* out_dev, int flags, gb_stream_t stream) {
  if (!pool) return GB_ERR_INVALID;
  if (!q_dev || !out_dev) return fail(pool, GB_ERR_INVALID, "decode: null pointer");
  if (flags < GB_PATH_AUTO || flags > GB_PATH_GROUPED) return fail(pool, GB_ERR_INVALID, "decode: bad flags");
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  gb_status st = append_layer(pool, layer, 1, k_new_dev, v_new_dev, s);
  if (st != GB_OK) return st;
  // Mode 1: shared-prefix segments go through the grouped tensor-core kernel and the
  // per-beam kernel reads only each beam's remainder; mode 0: every beam reads everything.
  // In mode 1 one attention kernel runs both: the grouped and the per-beam roles on their
  // shares of the SMs (decode_ctas), or one after the other on every SM.
  const int mode = (flags == GB_PATH_PER_BEAM || !pool->view.grouped) ? 0 : 1;
  prof_begin(pool, GB_PROF_ATTENTION, s);
  if (launch_decode(pool, layer, q_dev, scale, out_dev, mode, s) != cudaSuccess) return check_launch(pool, "decode");
  return check_launch(pool, "decode");
}

extern "C" gb_status gb_release(gb_pool* pool, const int32_t* slots_dev, int n, gb_stream_t stream) {
  if (!pool) return GB_ERR_INVALID;
  if (n < 0 || (n > 0 && !slots_dev)) return fail(pool, GB_ERR_INVALID, "release: bad arguments");
  if (pool->next_layer != 0) return fail(pool, GB_ERR_STATE, "release inside an open step");
  if (n == 0) return GB_OK;
  k_release<<<1, 1024, 0, reinterpret_cast<cudaStream_t>(stream)>>>(pool->view, slots_dev, n);
  pool->launches += 1;
  gb_status st = check_launch(pool, "release");
  if (st != GB_OK) return st;
  if (rebuild_segments(pool, reinterpret_cast<cudaStream_t>(stream)) != cudaSuccess)
    return check_launch(pool, "segments");
  return GB_OK;
}

extern "C" gb_status gb_pool_status(gb_pool* pool, int* device_status, gb_stream_t stream) {
  if (!pool || !device_status) return GB_ERR_INVALID;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  int v = 0;
  if (cudaMemcpyAsync(&v, pool->view.ctl + kCtlStatus, sizeof(int), cudaMemcpyDeviceToHost, s) != cudaSuccess ||
      cudaStreamSynchronize(s) != cudaSuccess)
    return check_launch(pool, "status");
  *device_status = v;
  return GB_OK;
}

extern "C" gb_status gb_pool_set_profile_events(gb_pool* pool, int which, void* start_event, void* stop_event) {
  if (!pool || which < 0 || which >= GB_PROF_SLOTS) return GB_ERR_INVALID;
  pool->prof_start[which] = static_cast<cudaEvent_t>(start_event);
  pool->prof_stop[which] = static_cast<cudaEvent_t>(stop_event);
  return GB_OK;
}

extern "C" gb_status gb_pool_read_step_stats(gb_pool* pool, int32_t* out, int max_steps, int* n_out,
                                             gb_stream_t stream) {
  if (!pool || !out || !n_out || max_steps < 0) return GB_ERR_INVALID;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  std::vector<int> ring((size_t)kStatsRing * kStatsWords);
  int steps = 0;
  if (cudaMemcpyAsync(&steps, pool->view.ctl + kCtlSteps, sizeof(int), cudaMemcpyDeviceToHost, s) != cudaSuccess ||
      cudaMemcpyAsync(ring.data(), pool->view.stats, ring.size() * sizeof(int), cudaMemcpyDeviceToHost, s) !=
          cudaSuccess ||
      cudaStreamSynchronize(s) != cudaSuccess)
    return check_launch(pool, "read_step_stats");
  const int n = std::min({max_steps, steps, kStatsRing});
  for (int i = 0; i < n; ++i) {
    const int step = steps - n + i;
    std::memcpy(out + (size_t)i * kStatsWords, ring.data() + (size_t)(step % kStatsRing) * kStatsWords,
                kStatsWords * sizeof(int));
  }
  *n_out = n;
  return GB_OK;
}

extern "C" gb_status gb_pool_launch_count(gb_pool* pool, uint64_t* count) {
  if (!pool || !count) return GB_ERR_INVALID;
  *count = pool->launches;
  return GB_OK;
}

extern "C" gb_status gb_pool_wait_selftest(gb_pool* pool, gb_stream_t stream) {
  if (!pool) return GB_ERR_INVALID;
  if (launch_wait_selftest(pool, reinterpret_cast<cudaStream_t>(stream)) != cudaSuccess)
    return check_launch(pool, "wait_selftest");
  pool->launches += 1;
  return check_launch(pool, "wait_selftest");
}

extern "C" gb_status gb_pool_clear_status(gb_pool* pool, gb_stream_t stream) {
  if (!pool) return GB_ERR_INVALID;
  k_clear_status<<<1, 1, 0, reinterpret_cast<cudaStream_t>(stream)>>>(pool->view);
  pool->launches += 1;
  return check_launch(pool, "clear_status");
}

extern "C" gb_status gb_pool_read_state(gb_pool* pool, const gb_pool_state* st, gb_stream_t stream) {
  if (!pool || !st) return GB_ERR_INVALID;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  const PoolView& v = pool->view;
  const size_t B = (size_t)v.max_beams;
  struct Copy { void* dst; const void* src; size_t bytes; } copies[] = {
      {st->tables, v.tables, B * v.max_pages * sizeof(int)},
      {st->seq_len, v.seq_len, B * sizeof(int)},
      {st->active, v.active, B * sizeof(int)},
      {st->gen, v.gen, B * sizeof(int)},
      {st->nsteps, v.nsteps, B * sizeof(int)},
      {st->mean, v.mean, B * sizeof(float)},
      {st->lineage, v.lineage, B * sizeof(unsigned)},
      {st->refcnt, v.refcnt, (size_t)v.num_pages * sizeof(int)},
      {st->free_bits, v.free_bits, (size_t)v.words * sizeof(unsigned)},
      {st->seg_cover, v.seg_cover, B * sizeof(int)},
      {st->seg_nseg, v.seg_nseg, B * sizeof(int)},
  };
  for (const Copy& c : copies) {
    if (!c.dst) continue;
    if (cudaMemcpyAsync(c.dst, c.src, c.bytes, cudaMemcpyDeviceToHost, s) != cudaSuccess)
      return check_launch(pool, "read_state");
  }
  if (cudaStreamSynchronize(s) != cudaSuccess) return check_launch(pool, "read_state");
  return GB_OK;
}
