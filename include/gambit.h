/*
 * gambit.h - C ABI of the GB300 (sm_103a) beam-decode library.
 *
 * The library implements the data-parallel hot path of thought-level beam
 * search ("Gambit", Algorithm 1): one decode step over a population of
 * reasoning beams that share forked KV-cache prefixes, the scorer probe at
 * thought boundaries, and the tournament's prune/branch, which keeps the
 * top-scoring beams and forks their block tables without copying KV.
 *
 * Conventions for every entry point
 * ---------------------------------
 * - Every function returns a gb_status; nothing throws across the ABI.
 *   gb_last_error() gives a short static description of the last host-side
 *   failure of a pool.
 * - Device work is enqueued asynchronously on the caller's stream
 *   (gb_stream_t is cudaStream_t; NULL means the legacy default stream).
 *   Host-side argument checks fail synchronously with GB_ERR_INVALID /
 *   GB_ERR_STATE / GB_ERR_UNSUPPORTED before anything is enqueued.
 * - Errors found on the device (out of pages, a bad slot id, a bounded wait
 *   that ran out) are recorded in a device status word: the first error
 *   sticks.  gb_pool_status() synchronises the stream and reads it.  A
 *   decode step whose page allocation failed does nothing: it changes no
 *   pool state and its attention outputs are zero.
 * - Ownership: the library never allocates device memory.  The caller
 *   allocates the KV pool and the metadata buffer (sizes from
 *   gb_pool_workspace_bytes), keeps them alive until gb_pool_destroy(), and
 *   frees them afterwards.  The opaque gb_pool handle is a small host
 *   struct owned by the library.
 * - Pointers named *_dev are device pointers; all others are host pointers.
 * - Slots: a pool has max_beams slots; a slot is active while it holds a
 *   beam.  Arrays indexed by slot have max_beams entries.
 * - GQA: query head h reads KV head h / (num_q_heads / num_kv_heads).
 */
#ifndef GAMBIT_H
#define GAMBIT_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef int gb_status;
#define GB_OK 0
#define GB_ERR_INVALID 1     /* bad argument or slot id */
#define GB_ERR_OOM 2         /* no free page (or a block table is full) */
#define GB_ERR_CUDA 3        /* a CUDA runtime call failed */
#define GB_ERR_STATE 4       /* call out of order (e.g. layers of a step, release of an inactive slot) */
#define GB_ERR_TIMEOUT 5     /* a bounded device-side wait ran out */
#define GB_ERR_UNSUPPORTED 6 /* shape/dtype combination without a kernel */

/* Element types. */
#define GB_F32 0
#define GB_BF16 1

/* Decode path selection for gb_decode_attention(). */
#define GB_PATH_AUTO 0      /* grouped tensor-core path where a shared segment is dense enough */
#define GB_PATH_PER_BEAM 1  /* every beam reads its whole context itself */
#define GB_PATH_GROUPED 2   /* like AUTO (kept for explicit requests) */

typedef struct CUstream_st* gb_stream_t; /* identical to cudaStream_t */
typedef struct gb_pool gb_pool;          /* opaque host handle */

typedef struct {
  int num_layers;          /* layers sharing one page id space (a page spans all layers) */
  int num_q_heads;         /* Hq */
  int num_kv_heads;        /* Hkv; Hq % Hkv == 0 */
  int head_dim;            /* D: 128 for GB_BF16, 64 for GB_F32 */
  int page_size;           /* P tokens per page: 16, 32 or 64 */
  int kv_dtype;            /* GB_F32 or GB_BF16: K/V storage and the query dtype */
  int64_t num_pages;       /* pages in the pool */
  int max_beams;           /* slots = capacity C of the tournament, <= 1024 */
  int max_pages_per_beam;  /* block-table width */
  int group_min_beams;     /* grouped path only for segments shared by >= this many beams (0: default 2) */
} gb_pool_config;

/* Host-side copies of the pool state, for tests and debugging (any member may be NULL). */
typedef struct {
  int32_t* tables;     /* [max_beams][max_pages_per_beam]; entries past ceil(seq_len/P) unspecified */
  int32_t* seq_len;    /* [max_beams] tokens in each slot's context (0 when inactive) */
  int32_t* active;     /* [max_beams] 1 when the slot holds a beam */
  int32_t* gen;        /* [max_beams] tokens generated since the beam's own creation */
  int32_t* nsteps;     /* [max_beams] scored thought steps n */
  float* mean;         /* [max_beams] running mean score s_bar */
  uint32_t* lineage;   /* [max_beams] unique id of the beam now in the slot */
  int32_t* refcnt;     /* [num_pages] active slots referencing each page */
  uint32_t* free_bits; /* [ceil(num_pages/32)] bit p%32 of word p/32 set when page p is free */
  int32_t* seg_cover;  /* [max_beams] leading full pages read by the grouped path (0 without it) */
  int32_t* seg_nseg;   /* [max_beams] shared-prefix segments covering them */
} gb_pool_state;

/*
 * Sizes of the two caller-allocated device buffers for a configuration.
 * kv_bytes: the paged KV pool, laid out [layer][page][K|V][kv_head][P][D] in
 * kv_dtype.  meta_bytes: block tables, refcounts, free bitmap, per-slot
 * scores, decode plans and split-KV partials.  Either output may be NULL.
 * Paged KV and block tables: Section 3.1 (branching "via prefix caching",
 * pruning "frees their non-shared KV-cache blocks").
 * Errors: GB_ERR_INVALID for an inconsistent config, GB_ERR_UNSUPPORTED for
 * a (kv_dtype, head_dim, Hq/Hkv) without a kernel.
 */
gb_status gb_pool_workspace_bytes(const gb_pool_config* cfg, size_t* kv_bytes, size_t* meta_bytes);

/*
 * Create a pool over caller memory.  kv_dev and meta_dev must be 256-byte
 * aligned and at least the sizes above.  The metadata is initialised on
 * `stream` (every page free, every slot inactive); K/V contents are left as
 * they are.  *out receives the handle.
 */
gb_status gb_pool_init(const gb_pool_config* cfg, void* kv_dev, void* meta_dev,
                       gb_stream_t stream, gb_pool** out);

/* Free the host handle (not the caller's device buffers). */
gb_status gb_pool_destroy(gb_pool* pool);

/*
 * Seed the C initial traces of Algorithm 1 ("S <- C initial traces from P"):
 * slots 0..n_beams-1 become active, all sharing the prompt's pages
 * (refcount n_beams each, lowest free page ids).  k_prompt_dev/v_prompt_dev:
 * [num_layers][prompt_len][Hkv][D] in kv_dtype.  Running means start at 0
 * with n = 0.  Slots get lineage ids in order.
 * Errors: GB_ERR_STATE unless every slot is inactive; GB_ERR_INVALID for a
 * bad count or length; out of pages is reported in the device status.
 */
gb_status gb_pool_seed(gb_pool* pool, int n_beams, int prompt_len, const void* k_prompt_dev,
                       const void* v_prompt_dev, gb_stream_t stream);

/*
 * One decode step of one layer for every active beam (Algorithm 1,
 * "Generate: advance one thought for all tau in S", one token at a time).
 * Appends k_new/v_new at each beam's next position, then computes GQA decode
 * attention over the beam's whole context through its block table:
 *   out[b][h] = sum_t softmax_t(scale * q[b][h] . K_b[t]) V_b[t]
 * where K_b/V_b are read from KV head h / G.  Layer 0 opens a step (reserves
 * the position for every beam, allocating the lowest free page at a page
 * boundary and copying a still-shared partial tail page); layers must then be
 * called in order 0..num_layers-1.
 *   q_dev:      [max_beams][Hq][D] in kv_dtype
 *   k_new_dev, v_new_dev: [max_beams][Hkv][D] in kv_dtype
 *   out_dev:    [max_beams][Hq][D] fp32 (rows of inactive slots are zero)
 *   flags:      GB_PATH_AUTO / GB_PATH_PER_BEAM / GB_PATH_GROUPED
 * Rows of inactive slots in the inputs are ignored.
 * Launches: the append, then one attention launch that also merges the
 * split and shared-prefix partial results into out_dev (bf16 pools; fp32
 * pools add a merge launch); layer 0 adds the step's planner first.  The
 * attention launch's CTAs wait (bounded) on each other's partial results, so
 * they must all get an SM within the wait limit (2 s): nothing else should
 * hold the GPU's SMs for that long meanwhile.
 * Errors: GB_ERR_STATE for a layer out of order; out of pages is reported in
 * the device status and makes the whole step a no-op; a wait that runs out
 * records GB_ERR_TIMEOUT and zeroes the outputs it could not complete.
 */
gb_status gb_decode_attention(gb_pool* pool, int layer, const void* q_dev, const void* k_new_dev,
                              const void* v_new_dev, float scale, float* out_dev, int flags,
                              gb_stream_t stream);

/*
 * Append n_tokens tokens to every active beam for one layer, without
 * attention (a chunk of a thought written at once).  Equivalent to n_tokens
 * decode steps' appends: page allocation follows the same order (token by
 * token, slots ascending).  k_dev/v_dev: [n_tokens][max_beams][Hkv][D].
 * Layer 0 reserves the positions; layers 1.. must follow in order.
 * Errors as gb_decode_attention.
 */
gb_status gb_append_kv(gb_pool* pool, int layer, int n_tokens, const void* k_dev,
                       const void* v_dev, gb_stream_t stream);

/*
 * Scorer probe at a thought boundary and the running-mean update of
 * Algorithm 1 ("s_bar <- s_bar + (f(h_n) - s_bar)/n"), with the probe
 * f(h) = sigmoid(w . h + bias) (Section 3.1 scores traces with a light-weight
 * scorer on the last-layer hidden state).
 *   hidden_dev:  [max_beams][hidden_dim] in hidden_dtype (GB_F32/GB_BF16)
 *   w_dev:       [hidden_dim] fp32
 *   boundary_mask_dev: [max_beams] u8, or NULL for every active slot; only
 *                masked active slots update (n += 1, s_bar updated in fp32:
 *                subtract, divide, add, each rounded)
 *   score_out_dev: [max_beams] fp32 probe score (0 for inactive slots), may be NULL
 * Errors: GB_ERR_INVALID unless hidden_dim is a positive multiple of 8.
 */
gb_status gb_score_probe(gb_pool* pool, const void* hidden_dev, int hidden_dtype, int hidden_dim,
                         const float* w_dev, float bias, const uint8_t* boundary_mask_dev,
                         float* score_out_dev, gb_stream_t stream);

/*
 * The same update with the two-layer MLP scorer (Section 4 evaluates Gambit with
 * a light-weight 2-layer MLP scorer; Section 3.1 admits any scorer of the
 * last-layer hidden state): f(h) = sigmoid(w2 . relu(W1 h + b1) + b2).  The
 * first layer runs on the tensor cores (bf16 in, fp32 accumulate).
 *   hidden_dev: [max_beams][hidden_dim] bf16, 16-byte aligned; hidden_dim a
 *               positive multiple of 64
 *   w1_dev:     [d_h][hidden_dim] bf16, 16-byte aligned
 *   b1_dev, w2_dev: [d_h] fp32; b2 the output bias
 *   boundary_mask_dev, score_out_dev: as gb_score_probe
 * Errors: GB_ERR_INVALID for bad sizes or alignment; GB_ERR_TOO_LARGE when
 * max_beams x d_h exceeds 5,242,880 (the pool's partial-sum buffer).
 */
gb_status gb_score_mlp(gb_pool* pool, const void* hidden_dev, int hidden_dim, const void* w1_dev,
                       const float* b1_dev, const float* w2_dev, float b2, int d_h,
                       const uint8_t* boundary_mask_dev, float* score_out_dev, gb_stream_t stream);

/*
 * Running-mean update with scores computed elsewhere (any scorer f_theta,
 * Section 3.1): for masked active slots, n += 1 and s_bar is updated exactly
 * as in gb_score_probe.  scores_dev: [max_beams] fp32; mask as above.
 */
gb_status gb_push_scores(gb_pool* pool, const float* scores_dev, const uint8_t* mask_dev,
                         gb_stream_t stream);

/*
 * One tournament round (Algorithm 1, Tournament; Eq. 2 and Eq. 3).
 * Active slots are ranked by s_bar descending (ties: lower slot first; NaN
 * last).  Eligible parents are active slots with gen >= warmup and, when
 * eligible_dev is given, eligible_dev[slot] != 0.
 *   Case 1 (fewer active slots than the capacity C, see gb_pool_set_capacity;
 *   default max_beams): the top min(C - active, |B|) eligible beams get one
 *   child each, placed in vacant slots ascending.
 *   Case 2 (C slots active): prune the bottom K_eff = min(K, (fanout-1) x
 *   eligible survivors) beams; each of the top eligible survivors gets
 *   fanout-1 children (the last one the remainder), placed in the pruned
 *   slots ascending.  fanout = 2 is Eq. 3 exactly.
 * A child gets its parent's block table (every page's refcount + 1; no KV is
 * copied), length, s_bar and n, gen = 0 and a new lineage id.  A pruned beam
 * drops its references; pages reaching refcount 0 become free.
 *   parent_out_dev:  [max_beams] int32: own slot for surviving beams, parent
 *                    slot for new children, -1 for inactive slots (may be NULL)
 *   pruned_out_dev:  [max_beams] u8: 1 where a beam was pruned (may be NULL)
 *   lineage_out_dev: [max_beams] u32 lineage ids after the round (may be NULL)
 * Errors: GB_ERR_INVALID for K < 0 or fanout < 2.
 */
gb_status gb_prune_branch(gb_pool* pool, int K, int fanout, int warmup, const uint8_t* eligible_dev,
                          int32_t* parent_out_dev, uint8_t* pruned_out_dev, uint32_t* lineage_out_dev,
                          gb_stream_t stream);

/*
 * The active slot the tournament would rank last (Algorithm 1, KV saturation: the trace with
 * the lowest running mean is evicted from the Scheduler view and kept in the Tree view as a
 * ghost, Section 3.2): NaN means rank last, then the lowest mean, ties to the higher slot -
 * the ranking of gb_prune_branch read from its end.  Writes the slot to *slot_out_dev (an
 * int32 device word), or -1 when no slot is active; the caller releases it with gb_release.
 * Errors: GB_ERR_INVALID for a null pointer.
 */
gb_status gb_pool_last_ranked(gb_pool* pool, int32_t* slot_out_dev, gb_stream_t stream);

/*
 * The tree's capacity C (Algorithm 1's C; Section 3.2, Tree view): the
 * tournament takes Case 1 while fewer than C traces are active and Case 2
 * otherwise, and Case 1 never grows the active set beyond C.  Default and
 * maximum: max_beams.  A caller that evicts a trace as a ghost (it keeps its
 * place in the Tree view but no longer runs, Section 3.2) lowers C by one so
 * that the ghost still counts against the capacity.  Host-side setting, read
 * by the next gb_prune_branch calls.  Errors: GB_ERR_INVALID unless
 * 1 <= capacity <= max_beams.
 */
gb_status gb_pool_set_capacity(gb_pool* pool, int capacity);

/*
 * Release slots whose traces completed ("move completed traces to F") or
 * were evicted as ghost traces (Section 3.2): each listed slot drops its page
 * references (pages reaching 0 become free) and becomes inactive.  slots_dev:
 * [n] int32 device array, processed in order.  A slot out of range records
 * GB_ERR_INVALID, an inactive slot GB_ERR_STATE, in the device status; the
 * entry is skipped.
 */
gb_status gb_release(gb_pool* pool, const int32_t* slots_dev, int n, gb_stream_t stream);

/* Synchronise `stream` and read the device status word (GB_OK or the first error). */
gb_status gb_pool_status(gb_pool* pool, int* device_status, gb_stream_t stream);

/* Reset the device status word to GB_OK (enqueued on `stream`). */
gb_status gb_pool_clear_status(gb_pool* pool, gb_stream_t stream);

/*
 * Diagnostic of the failure path (not part of the method): enqueue one warp
 * that waits, with the attention launch's bounded wait, for a (beam, KV head)
 * record count that no kernel raises.  After the wait limit (2 s) it records
 * GB_ERR_TIMEOUT in the device status and returns, leaving the context and the
 * pool usable (clear the status to go on).  It touches no pool state but the
 * status word; it must not overlap a decode step of the pool.
 */
gb_status gb_pool_wait_selftest(gb_pool* pool, gb_stream_t stream);

/* Synchronise `stream` and copy the pool state into host arrays (see gb_pool_state). */
gb_status gb_pool_read_state(gb_pool* pool, const gb_pool_state* state, gb_stream_t stream);

/*
 * Instrumentation (not part of the method).  Record caller-created CUDA
 * events (cudaEvent_t) immediately before and after one kernel of the
 * following calls on this pool, so a caller can time that kernel alone on its
 * own stream: `which` is GB_PROF_DECODE (the attention launch of gb_decode_attention),
 * GB_PROF_PROBE (gb_score_probe, gb_score_mlp, or all of gb_scorer_step), GB_PROF_PRUNE
 * (all of gb_prune_branch or gb_fork_slots, the shared-prefix segment rebuild included),
 * GB_PROF_GROUPED (the attention launch when it has the grouped shared-prefix role),
 * GB_PROF_PLAN (the step planner: page allocation and decode plans, layer 0),
 * GB_PROF_APPEND (the K/V append of a layer), GB_PROF_COMBINE (the separate merge of
 * partial results after the fp32 kernel; bf16 pools merge inside the attention launch) or
 * GB_PROF_ATTENTION (the attention of a layer, up to its merged output except for the fp32
 * kernel's separate merge).  Passing NULL events stops recording.  The events stay
 * owned by the caller.  Under stream capture the records become external event
 * nodes of the graph.
 */
#define GB_PROF_DECODE 0
#define GB_PROF_PROBE 1
#define GB_PROF_PRUNE 2
#define GB_PROF_GROUPED 3
#define GB_PROF_PLAN 4
#define GB_PROF_APPEND 5
#define GB_PROF_COMBINE 6
#define GB_PROF_ATTENTION 7
#define GB_PROF_SLOTS 8
gb_status gb_pool_set_profile_events(gb_pool* pool, int which, void* start_event, void* stop_event);

/*
 * Work accounting of the most recent decode/append steps (not part of the method).
 * Synchronises `stream` and copies up to max_steps records, oldest first, into
 * out[n][10] (host): [0] tokens per KV head the per-beam path reads when every
 * beam reads its whole context, [1] the same with shared-prefix segments taken
 * by the grouped path, [2] sum over segments of (query rows of one KV head) x
 * tokens, [3] sum over segments of (128-row tiles) x tokens, [4] segments,
 * [5] 128-row tiles, [6] tokens appended by the step, [7] step index,
 * [8] sum over segments of their tokens (shared tokens per KV head, each once),
 * [9] active beams.
 * *n_out receives the number of records (at most the last 4096 steps are kept).
 */
gb_status gb_pool_read_step_stats(gb_pool* pool, int32_t* out, int max_steps, int* n_out, gb_stream_t stream);

/* Number of kernels this pool has launched since gb_pool_init (host-side count). */
gb_status gb_pool_launch_count(gb_pool* pool, uint64_t* count);

/*
 * Decode attention over caller-managed pages that allocates nothing.
 *
 * The paper has no counterpart; this entry point exists for callers that cannot
 * allocate device memory where they decode - for example a serving process whose
 * allocator takes the GPU's memory when it starts and allows no allocation on the
 * token path, or code running inside a framework whose device memory it does not
 * own.  The caller passes only inputs and outputs; the call's working memory (work
 * plan and split-KV partial results) is a fixed 32 MiB array in the library's own
 * device memory, which every GPU that loads the library holds until the process
 * exits.  No cudaMalloc, cudaFree or allocating library routine is called.
 *
 * Computes, for every row b with seq_len[b] > 0 and query head h,
 *   out[b][h] = sum_t softmax_t(scale * q[b][h] . K_b[t]) V_b[t],  t in [0, seq_len[b])
 * where token t of row b is row t % page_size of page tables[b][t / page_size] and
 * query head h reads KV head h / (num_q_heads / num_kv_heads).  Rows with
 * seq_len[b] == 0 give zeros.  Arguments (device pointers):
 *   kv:      one layer's pages, [num_pages][K|V][num_kv_heads][page_size][head_dim] in
 *            kv_dtype (the layout of a gb_pool layer), 16-byte aligned
 *   tables:  int32 [num_beams][max_pages_per_beam];  seq_len: int32 [num_beams]
 *   q:       [num_beams][num_q_heads][head_dim] in kv_dtype, 16-byte aligned
 *   out:     fp32 [num_beams][num_q_heads][head_dim]
 * Rows must satisfy 0 <= seq_len[b] <= max_pages_per_beam * page_size: a row outside
 * that range is not read (its output is zero) and the call's device status records
 * GB_ERR_INVALID.  Page ids are checked too: an id outside [0, num_pages) is not
 * dereferenced (page 0 is read in its place), that row's output is unspecified and the
 * status records GB_ERR_INVALID.  A bounded device-side wait that runs out records
 * GB_ERR_TIMEOUT.  gb_paged_decode_noalloc_status() reads that status word.
 *
 * The scratch array is shared by every call on a device and keeps the last call's
 * contents; each call rewrites all of it that it reads, and clears its own status
 * word first.  Calls whose GPU work overlaps (different streams, or host threads issuing
 * concurrently) race on it: keep them ordered, e.g. on one stream.
 * The first call on a device looks up the array's device address with
 * cudaGetSymbolAddress (with that device current); that first call should come
 * before any stream capture.
 * Errors: GB_ERR_INVALID for bad shapes or null/misaligned pointers, or when
 * num_beams x ceil(max_pages_per_beam x page_size / 16) x num_kv_heads reaches 2^31,
 * GB_ERR_UNSUPPORTED for a (kv_dtype, head_dim, Hq/Hkv) without a kernel, and
 * GB_ERR_TOO_LARGE when the scratch needed, 256-byte rounded
 *   128 + 4*num_beams + 12*(num_beams+1) + 4*(W + num_beams*num_kv_heads)*G*(head_dim+2)
 * bytes with W = 8 x (multiprocessor count) and G = num_q_heads/num_kv_heads, exceeds 32 MiB
 * (for G = 4, head_dim 128 and 8 KV heads: up to 1024 rows on a 152-SM GB300).
 */
#define GB_ERR_TOO_LARGE 7  /* the call needs more fixed scratch than the library holds */
typedef struct {
  const void* kv;
  const int32_t* tables;
  const int32_t* seq_len;
  const void* q;
  float* out;
  int num_beams;
  int num_q_heads;
  int num_kv_heads;
  int head_dim;
  int page_size;
  int kv_dtype;
  int max_pages_per_beam;
  int64_t num_pages;
  float scale;
} gb_paged_decode_args;
gb_status gb_paged_decode_noalloc(const gb_paged_decode_args* args, gb_stream_t stream);

/*
 * Device status of the most recent gb_paged_decode_noalloc() call on the current device
 * (GB_OK, or the first error its kernels recorded: GB_ERR_INVALID for a row length or
 * page id out of range, GB_ERR_TIMEOUT for a bounded wait that ran out).  Synchronises
 * `stream` (pass the stream of that call) and copies the status word of the library's
 * scratch array into *device_status with one cudaMemcpyAsync; allocates nothing.  The
 * paper has no counterpart: it belongs to the allocation-free entry point above.
 */
gb_status gb_paged_decode_noalloc_status(int* device_status, gb_stream_t stream);

/*
 * Apply a tournament decided on another pool (for example the generator's pool's
 * gb_prune_branch parent_out) to this pool: every slot s with parent_of[s] >= 0 and
 * parent_of[s] != s becomes a child of slot parent_of[s] - it drops its own page
 * references (pages reaching 0 become free), takes the parent's block table (every
 * page's refcount + 1; nothing is copied), length, s_bar and n, gen = 0 and a new
 * lineage id (children in ascending slot order).  Other slots are unchanged.
 * Section 3.1: a branched trace continues from its parent's state via prefix
 * caching; this keeps a second per-trace cache (the sequence scorer's) in step.
 *   parent_of_dev: [max_beams] int32 device array; a parent must keep
 *                  parent_of[parent] = parent (survivors), and be active.
 * A parent id >= max_beams records GB_ERR_INVALID in the device status.
 * Errors: GB_ERR_STATE for an unseeded pool or inside an open step.
 */
gb_status gb_fork_slots(gb_pool* pool, const int32_t* parent_of_dev, gb_stream_t stream);

/*
 * The history-aware sequence scorer (Appendix, "Evaluating Search Generalization",
 * Eq. 4-6), run incrementally: for each trace's step hidden states h_1 .. h_t,
 *   x_t = GELU(W_in LN(h_t)),  z_1..z_t = SequenceTransformer(x_1..x_t),
 *   y_t = sigmoid(w_out . LN(z_t) + b_out).
 * The transformer has L pre-norm layers: causal multi-head attention with rotary
 * embeddings (pairs (i, i + 64), angle t * 10000^(-i/64)), Hq query heads over Hkv
 * key/value heads of 128 dims, then a SwiGLU FFN (W_2 (SiLU(W_1 u) * W_3 u)).
 * LayerNorms have gain and bias, eps 1e-5; GELU is the erf form; d_model = Hq * 128.
 *
 * The scorer's key/value cache is a second gb_pool, the step pool, holding one token
 * per thought step: num_layers = L, num_q_heads = Hq, num_kv_heads = Hkv, head_dim
 * 128, kv_dtype GB_BF16, max_beams = the generator pool's.  Position 0 of every
 * trace is the hidden state at the end of the shared prompt (gb_scorer_seed); each
 * thought boundary adds one position (gb_scorer_step).  Branching and pruning are
 * mirrored with gb_fork_slots and gb_release on the step pool.  Matrix products run
 * on the tensor cores (bf16 operands, fp32 accumulation); the residual stream is fp32.
 *
 * Weights: one device buffer, 256-byte aligned, holding these tensors at the offsets
 * gb_scorer_sizes reports (row-major; "f32" fp32, "bf16" bfloat16):
 *   0 ln_in gain f32[H], 1 ln_in bias f32[H], 2 W_in bf16[d][H],
 *   per layer l (base 3 + 8 l): ln1 gain f32[d], ln1 bias f32[d],
 *     W_qkv bf16[(Hq + 2 Hkv) 128][d] (q heads, then k heads, then v heads),
 *     W_o bf16[d][d], ln2 gain f32[d], ln2 bias f32[d],
 *     W_13 bf16[2F][d] (the F rows of W_1, then the F rows of W_3), W_2 bf16[d][F],
 *   then (base 3 + 8 L): ln_out gain f32[d], ln_out bias f32[d], w_out f32[d], b_out f32[1].
 * Workspace: one device buffer, 256-byte aligned, of the size gb_scorer_sizes reports;
 * the caller owns both buffers.  Calls using one workspace must be ordered (one stream).
 */
typedef struct {
  int hidden_dim;  /* H: the generator's hidden size (positive multiple of 64) */
  int ffn_dim;     /* F: SwiGLU inner size (positive multiple of 64) */
} gb_scorer_config;

/*
 * Sizes of the weight buffer and the workspace for a step pool, and the byte offset
 * of each weight tensor (offsets[0 .. *n_offsets), in the order above; offsets may be
 * NULL, otherwise max_offsets must be >= 3 + 8 L + 4).  Any output may be NULL.
 * Errors: GB_ERR_UNSUPPORTED for a step pool or sizes the scorer cannot run on (not
 * bf16 with 128-dim heads, H or F not multiples of 64, more than 64 layers).
 */
gb_status gb_scorer_sizes(gb_pool* step_pool, const gb_scorer_config* cfg, size_t* weight_bytes,
                          size_t* workspace_bytes, size_t* offsets, int max_offsets, int* n_offsets);

/*
 * Position 0: run the layer stack on h0_dev (bf16 [H], the hidden state at the end of
 * the prompt) and seed the step pool's slots 0..n_beams-1 with its per-layer keys and
 * values (gb_pool_seed with a one-token prompt).
 * Errors: GB_ERR_STATE if the step pool is already seeded, GB_ERR_INVALID for bad
 * pointers, alignment or count, plus gb_pool_seed's.
 */
gb_status gb_scorer_seed(gb_pool* step_pool, const gb_scorer_config* cfg, const void* weights_dev,
                         void* workspace_dev, const void* h0_dev, int n_beams, gb_stream_t stream);

/*
 * One thought boundary for every active slot of the step pool: hidden_dev is bf16
 * [max_beams][H] (16-byte aligned; rows of inactive slots are ignored), the new
 * position's key/value is appended to each trace's history and
 *   score_out_dev[s] = y_t (Eq. 6) of slot s, 0 for inactive slots (fp32 [max_beams]).
 * Feed the scores to the generator pool's running means with gb_push_scores.
 * Errors: GB_ERR_STATE for an unseeded step pool or an open step; out of pages in
 * the step pool is reported in its device status (the scores are then invalid).
 */
gb_status gb_scorer_step(gb_pool* step_pool, const gb_scorer_config* cfg, const void* weights_dev,
                         void* workspace_dev, const void* hidden_dev, float* score_out_dev,
                         gb_stream_t stream);

/* Short description of the pool's last host-side failure ("" if none); static storage. */
const char* gb_last_error(gb_pool* pool);

#ifdef __cplusplus
}
#endif
#endif /* GAMBIT_H */
