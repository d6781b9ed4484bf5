// Internal definitions shared by the library's translation units.
#pragma once

#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <stdint.h>
#include <string>
#include <utility>

#include "gambit.h"

namespace gb {

constexpr int kMaxBeams = 1024;    // slots per pool (one thread per slot in the planners)
constexpr int kChunk = 16;         // tokens per split-KV work unit (a page is 1..4 chunks)
constexpr int kDecodeWarps = 8;    // warps per CTA of the split-KV decode kernel (one CTA per SM)
constexpr int kDecodeStages = 3;   // TMA ring depth per warp
constexpr int kDecodeCtasPerSm = 1;
constexpr int kMaxDecodeWarps = 4096;
#ifndef GB_MMA_WARPS
#define GB_MMA_WARPS 12  // warps per CTA of the warp-MMA per-beam kernel (one CTA per SM)
#endif
constexpr int kMmaWarps = GB_MMA_WARPS;
constexpr int kMaxCowJobs = 1024;
constexpr int kMaxSegDepth = 16;
constexpr int kMaxSegRecords = 48;  // grouped partial records per beam (segments x token splits)
constexpr int kStatsRing = 4096;   // steps kept in the step-stats ring
constexpr int kStatsWords = 10;  // words per step record of the step-stats ring
constexpr int kMlpScratchFloats = 320 * 128 * 128;  // K-split partials of the MLP scorer's first layer (20 MiB)

// Control words at the start of the metadata buffer.
enum Ctl : int {
  kCtlStatus = 0,      // first device-side error (GB_OK when none)
  kCtlStepOk = 1,      // 1 while the current decode step has its pages
  kCtlDone = 2,        // last-CTA-done ticket counter (reset by the last CTA)
  kCtlCursor = 3,      // lowest free-bitmap word that may hold a free page
  kCtlNextLineage = 4, // next lineage id to hand out
  kCtlFree = 5,        // number of free pages
  kCtlCowJobs = 6,     // copy-on-write jobs of the open step (rows copied by each layer's append)
  kCtlSegCount = 7,    // shared-prefix segments found by the last rebuild
  kCtlSegMembers = 8,  // (beam, depth) memberships handed out by the last rebuild
  kCtlSegTiles = 9,    // 128-row query tiles over all segments
  kCtlSegRowTok = 10,  // sum over segments of (query rows of one KV head) x tokens
  kCtlSegTileTok = 11, // sum over segments of (128-row tiles) x tokens
  kCtlSteps = 12,      // steps opened so far (index into the step-stats ring)
  kCtlSegSplit = 13,   // tokens per grouped work unit (segments are split along tokens)
  kCtlGrpNext = 14,    // next grouped work unit to hand out (zeroed by k_append)
  kCtlGrpDone = 15,    // grouped-role CTAs finished (zeroed by k_append)
  kCtlSegTok = 16,     // sum over segments of their tokens (the shared tokens the grouped path reads once)
  kCtlBarCount = 17,   // grid-barrier arrivals of the tournament kernel (only grows)
  kCtlSegGen = 19,     // segment rebuilds so far (stamps the per-page claim words)
  kCtlSegAlloc = 20,   // words 20-21: (segments << 32 | member slots) handed out by the running rebuild
  kCtlTailShared = 22, // 1 when a partial tail page may be shared (set by seed and forks, cleared by the planner)
  kCtlPairNext = 23,   // next (beam, KV head) pair to merge in the attention launch (zeroed by k_append)
  kCtlWords = 32
};

// Byte offsets of the metadata regions.
struct MetaLayout {
  size_t ctl, tables, seq_len, active, gen, nsteps, mean, lineage, refcnt, free_bits;
  size_t plan, cow, partials, total, stats;
  // shared-prefix segments
  size_t seg_cover, seg_nseg, seg_owner, seg_i0, seg_len, seg_rep, seg_g, seg_mem_off, seg_fill, seg_members,
      seg_tile_seg, seg_tile_t, grec, seg_bid, seg_rec_off, seg_nrec, seg_splits, seg_tile_split, seg_hist, pair_cnt;
  int words;            // free-bitmap words
  size_t mlp_scratch;   // MLP scorer partial sums
  int partial_records;  // split-KV partial records
  int record_floats;    // floats per partial record: G*(D+2)
};

MetaLayout meta_layout(const gb_pool_config& c);

// Plain-old-data view of a pool passed by value to kernels.
struct PoolView {
  int layers, Hq, Hkv, D, P, G, dtype, esize, max_beams, max_pages, words;
  long long num_pages;
  char* kv;             // KV pool base
  long long page_elems; // elements of one (layer, page): 2*Hkv*P*D
  int* ctl;
  int* tables;          // [max_beams][max_pages]
  int* seq_len;
  int* active;
  int* gen;
  int* nsteps;
  float* mean;
  unsigned* lineage;
  int* refcnt;
  unsigned* free_bits;
  int* plan;            // [2 modes][3][max_beams + 1]: offsets, chunk counts, start tokens
  int* cow;             // [kMaxCowJobs][3] (old page, new page, rows) of the open step's copy-on-writes
  // Shared-prefix segments (rebuilt after seed, prune/branch and release):
  int grouped;          // 1 when the grouped tensor-core path exists for this pool's dtype/shape
  int group_min;        // segments need at least this many sharing beams
  int* seg_cover;       // [max_beams] leading full pages of the beam covered by segments
  int* seg_nseg;        // [max_beams] segments the beam belongs to (by depth)
  unsigned long long* seg_owner;  // [num_pages] claim word of a segment-start page: (rebuild gen << 32) | (segment id + 1)
  int* seg_i0;          // [segments] first table index
  int* seg_len;         // [segments] pages
  int* seg_rep;         // [segments] a member beam whose table lists the pages
  int* seg_g;           // [segments] member beams
  int* seg_mem_off;     // [segments] offset of its members
  int* seg_fill;        // [segments] members written so far
  int* seg_members;     // [memberships] beam * kMaxSegDepth + depth
  int* seg_tile_seg;    // [tiles] segment of each 128-row query tile
  int* seg_tile_t;      // [tiles] tile index within the segment
  int* seg_tile_split;  // [tiles] token split of the unit
  int* seg_splits;      // [segments] token splits of the segment
  int* seg_bid;         // [max_beams][kMaxSegDepth] segment id of the beam's k-th segment
  int* seg_rec_off;     // [max_beams][kMaxSegDepth] first grouped record of that segment
  int* seg_nrec;        // [max_beams] grouped records of the beam
  int* seg_hist;        // [2][256] work units per length bucket, and units placed per bucket (rebuild scratch)
  int num_sms;          // multiprocessors (sizes the grouped work split)
  float* grec;          // [max_beams][kMaxSegDepth][Hkv] grouped partial records
  int* stats;           // [kStatsRing][kStatsWords] work of recent steps (see gb_pool_read_step_stats)
  float* partials;
  int* pair_cnt;        // [max_beams * Hkv] per-beam records written for each (beam, KV head) by the
                        // running attention launch (zeroed by k_append before it)
  int record_floats;
  float* mlp_scratch;   // [kMlpScratchFloats] K-split partials of the MLP scorer
};

// Plan arrays: mode 0 = per-beam only, mode 1 = with grouped coverage.
__host__ __device__ inline int* plan_off(const PoolView& v, int mode) {
  return v.plan + (size_t)mode * 3 * (v.max_beams + 1);
}
__host__ __device__ inline int* plan_n(const PoolView& v, int mode) {
  return plan_off(v, mode) + (v.max_beams + 1);
}
__host__ __device__ inline int* plan_start(const PoolView& v, int mode) {
  return plan_off(v, mode) + 2 * (v.max_beams + 1);
}

#ifndef GB_DECODE_WEIGHT
#define GB_DECODE_WEIGHT 45  // relative cost of a per-beam token against a grouped tile token (percent)
#endif

#ifndef GB_SPLIT_BYTES_PER_SM
#define GB_SPLIT_BYTES_PER_SM (8ll << 20)
#endif

// A mode-1 step launches one attention kernel with a grouped and a per-beam role.  When the
// step's attention reads little per SM (below GB_SPLIT_BYTES_PER_SM), both roles are
// latency-bound and run side by side, each on its own share of the CTAs (one per SM): the
// per-beam role takes decode_ctas(v, grid) of them, in proportion to its (16-token chunk x
// KV head) tokens against the grouped role's (128-row tile x token) work per KV head, and
// the grouped role the rest.  Otherwise every CTA runs the grouped role and then the
// per-beam role.  The kernel and the combine compute the same split from the step's plan.
__device__ __forceinline__ int decode_ctas(const PoolView& v, int grid);

// Element offset of row `row` of the K (kv=0) or V (kv=1) slab of (layer, page, head).
__device__ __forceinline__ long long kv_elem_offset(const PoolView& v, int layer, long long page,
                                                    int kv, int head, int row) {
  return ((((long long)layer * v.num_pages + page) * 2 + kv) * v.Hkv + head) * (long long)v.P * v.D +
         (long long)row * v.D;
}

// Programmatic dependent launch.  Every kernel of the library begins with pdl_wait(),
// before any global memory access: launched normally it returns at once; launched with
// programmatic stream serialization (launch_pdl) the kernel may be scheduled while the
// previous kernel in the stream is still running, and pdl_wait() blocks until that
// kernel has completed and its writes are visible - the same ordering as a plain launch,
// without the gap between the two kernels.  pdl_launch_dependents() lets the next
// kernel be scheduled as soon as every CTA of this one has started.
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_launch_dependents() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

__device__ __forceinline__ bool split_sms(const PoolView& v, long long td, long long tg) {
  const long long bytes = (td + tg) * 2 * v.D * v.esize;
  return td > 0 && tg > 0 && bytes < GB_SPLIT_BYTES_PER_SM * v.num_sms;
}
__device__ __forceinline__ int decode_ctas(const PoolView& v, int grid) {
  const long long td = (long long)plan_off(v, 1)[v.max_beams] * kChunk;  // tokens x KV heads
  const long long tg = (long long)v.ctl[kCtlSegTileTok] * v.Hkv;
  if (!split_sms(v, td, tg)) return grid;
  const long long wd = td * GB_DECODE_WEIGHT, wg = tg * 100;
  const long long n = (wd * grid + (wd + wg) / 2) / (wd + wg);
  return (int)(n < 1 ? 1 : (n > grid - 1 ? grid - 1 : n));
}

__device__ __forceinline__ void set_status(int* ctl, int code) {
  atomicCAS(&ctl[kCtlStatus], GB_OK, code);
}

// Mark page p free (bitmap, allocation cursor, free count).
__device__ __forceinline__ void mark_free(const PoolView& v, int p) {
  atomicOr(&v.free_bits[p >> 5], 1u << (p & 31));
  atomicMin(&v.ctl[kCtlCursor], p >> 5);
  atomicAdd(&v.ctl[kCtlFree], 1);
}

// Drop one reference to page p; frees it when the count reaches zero.
__device__ __forceinline__ void unref_page(const PoolView& v, int p) {
  if (atomicSub(&v.refcnt[p], 1) == 1) mark_free(v, p);
}

// Block-wide exclusive scan of one int per thread (blockDim.x <= 1024, multiple of 32).
// `tmp` must hold 33 ints of shared memory.  Returns the exclusive prefix; *total gets the sum.
__device__ __forceinline__ int block_exclusive_scan(int x, int* tmp, int* total) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nwarps = blockDim.x >> 5;
  int inc = x;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    int y = __shfl_up_sync(0xffffffffu, inc, o);
    if (lane >= o) inc += y;
  }
  if (lane == 31) tmp[warp] = inc;
  __syncthreads();
  if (warp == 0) {
    int w = lane < nwarps ? tmp[lane] : 0;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      int y = __shfl_up_sync(0xffffffffu, w, o);
      if (lane >= o) w += y;
    }
    if (lane < nwarps) tmp[lane] = w;  // inclusive warp totals
    if (lane == nwarps - 1) tmp[32] = w;
  }
  __syncthreads();
  int r = inc - x + (warp > 0 ? tmp[warp - 1] : 0);
  *total = tmp[32];
  __syncthreads();
  return r;
}

// Host side --------------------------------------------------------------------

// Launch with programmatic stream serialization (see pdl_wait).  Built with -DGB_NO_PDL
// it is a plain launch.
template <typename... KArgs, typename... Args>
inline cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t s,
                              Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
#ifndef GB_NO_PDL
  cfg.attrs = attr;
  cfg.numAttrs = 1;
#endif
  return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}

struct DecodeShape {
  int dtype, D, G;
};
bool decode_supported(int dtype, int D, int G);

}  // namespace gb

// The opaque host handle.
struct gb_pool {
  gb_pool_config cfg;
  gb::MetaLayout layout;
  gb::PoolView view;
  int device;
  int num_sms;
  int decode_warps;   // warps launched by the split-KV decode kernel
  int next_layer;     // layer expected by the next decode/append call (0 opens a step)
  int step_tokens;    // tokens reserved by the open step
  bool seeded;
  int group_min;
  int capacity = 0;   // the tree's capacity C for the tournament (0: max_beams)
  alignas(64) unsigned char tmap[128];      // CUtensorMap over the KV pool (grouped path)
  bool have_tmap = false;
  alignas(64) unsigned char dtmap[128];     // CUtensorMap over the KV pool (per-beam bf16 path)
  alignas(64) unsigned char dtmap_half[128];  // the same with an 8-token box (short tail chunks)
  bool have_dtmap = false;
  int tmap_oob = 0;                          // first row group past the tensor map (loads zeros)
  std::string last_error;
  unsigned long long launches = 0;          // kernels launched by this pool
  cudaEvent_t prof_start[GB_PROF_SLOTS] = {};  // caller-owned instrumentation events
  cudaEvent_t prof_stop[GB_PROF_SLOTS] = {};
};

namespace gb {
gb_status fail(gb_pool* pool, gb_status code, const char* what);

// Instrumentation: record the caller's event pair around one kernel, if set.  Under
// stream capture the records become external event nodes, so the events are recorded
// (and can be timed) each time the graph runs.
inline void prof_record(cudaEvent_t e, cudaStream_t s) {
  cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
  cudaStreamIsCapturing(s, &cs);
  cudaEventRecordWithFlags(e, s, cs == cudaStreamCaptureStatusActive ? cudaEventRecordExternal : cudaEventRecordDefault);
}
inline void prof_begin(gb_pool* p, int which, cudaStream_t s) {
  if (p->prof_start[which]) prof_record(p->prof_start[which], s);
}
inline void prof_end(gb_pool* p, int which, cudaStream_t s) {
  if (p->prof_stop[which]) prof_record(p->prof_stop[which], s);
}
gb_status check_launch(gb_pool* pool, const char* what);
// Raise a kernel's dynamic shared memory limit to `bytes` on the current device.  The
// attribute belongs to the device, so it is set once per (kernel, device), under a lock.
cudaError_t set_max_dynamic_smem(const void* kernel, int bytes);


// Kernel launchers implemented in the other translation units.
// The attention of one layer-step on s, written to out: mode 0, the per-beam kernel; mode 1,
// the attention kernel with the grouped and per-beam roles (launch_attention).  The bf16
// kernels merge their records themselves; the fp32 kernel is followed by k_combine.
cudaError_t launch_decode(gb_pool* pool, int layer, const void* q, float scale, float* out, int mode,
                          cudaStream_t s);
cudaError_t launch_decode_view(const PoolView& v, int W, int layer, const void* q, float scale, float* out,
                               cudaStream_t s);
cudaError_t rebuild_segments(gb_pool* pool, cudaStream_t s);
cudaError_t launch_attention(gb_pool* pool, int layer, const void* q, float scale, float* out, cudaStream_t s);
cudaError_t launch_wait_selftest(gb_pool* pool, cudaStream_t s);
void make_kv_tensor_maps(gb_pool* pool);
cudaError_t launch_probe(gb_pool* pool, const void* hidden, int hidden_dtype, int H, const float* w,
                         float bias, const uint8_t* mask, float* score_out, const float* scores_in,
                         cudaStream_t s);
// Split-K bf16 GEMM on the tensor cores (gemm.cu): P[s][m][n] over k-range s of A[m][k] B[n][k].
int gemm_splits(int M, int N, int K, int num_sms, size_t max_floats);
cudaError_t gemm_partials(const void* A, int M, const void* B, int N, int K, int splits, float* P, int* ctl,
                          cudaStream_t s);
cudaError_t launch_mlp(gb_pool* pool, const void* hidden, int H, const void* w1, const float* b1, const float* w2,
                       float b2, int dh, const uint8_t* mask, float* score_out, cudaStream_t s);
cudaError_t launch_prune_branch(gb_pool* pool, int K, int fanout, int warmup, const uint8_t* elig,
                                int32_t* parent_out, uint8_t* pruned_out, uint32_t* lineage_out,
                                cudaStream_t s);
}  // namespace gb
