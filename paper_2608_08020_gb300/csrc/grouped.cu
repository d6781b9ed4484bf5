// Grouped shared-prefix decode attention on tcgen05 tensor cores.
//
// For a segment of pages shared by g beams, the g x G query rows of one KV head
// (G = Hq / Hkv) are stacked into one 128-row tile, so the segment's K and V are
// read once for all of them and Q.K^T and P.V become dense contractions:
//   S[128 x 128]  = Q[128 x 128] . K_tile^T               (tcgen05.mma kind::f16, fp32 in TMEM)
//   O[128 x 128] += P_0[128 x 64] . V_0 + P_1[128 x 64] . V_1  (the tile's two 64-token halves)
// over 128-token tiles.  A unit of work is (segment, KV head, 128-row query tile, token
// split); a persistent grid of one CTA per SM walks the flat unit list, and the tiles of
// all of a CTA's units form one continuous pipeline.
//
// Warp roles (352 of the attention kernel's 384 threads; the last warp idles in this role):
//   warps 0-3  softmax group 0 and warps 4-7 softmax group 1: thread r of group k owns
//              query row r (TMEM lane r) and tokens [64k, 64k + 64) of every tile.  Each
//              tile the two groups swap their row maxima through shared memory, so both
//              keep the same running max m and their P.V products add into one
//              accumulator O; each keeps its own sum l_k and writes P_k (bf16) over the
//              first 32 of its S columns.  At the end of a unit the groups add their
//              sums and each writes half of the unnormalised record (m, l, o) of its row;
//   warp 8     K producer: takes the next unit from the grid-wide counter (the work list
//              is sorted longest first, so this is longest-processing-time-first across
//              the CTAs), publishes it to the other roles through a 4-slot ring,
//              gathers the unit's query rows into the Q buffer and streams the K half
//              of every tile through a 3-stage ring, one 5D TMA per page, issued by
//              several lanes at once;
//   warp 10    V producer: follows the same units and streams the V halves through a
//              second 3-stage ring.  A K slot is free once S has read it, long before
//              P.V has read the tile's V, so K runs further ahead than a joint K/V
//              stage would let it;
//   warp 9     MMA issuer: polls and issues S(n+1) or P.V(n), whichever is ready first;
//              P.V takes P straight from tensor memory.
// Handshakes are mbarriers: full/empty per K stage and per V stage, sched_full/sched_empty
// per unit slot, q_full/q_empty, s_full, p_full and pv_done per S/P tile (three in
// tensor memory), max_full per tile parity, xch_full and o_free per unit.  The grid-wide
// work counter is zeroed by k_append before each launch.  An S/P buffer is reused by
// S(n+3) only after P.V(n) has been issued: the tensor core runs a CTA's MMAs in issue
// order, so P(n) has been read before S(n+3) overwrites it.  With three buffers S runs two
// tiles ahead of the softmax.
//
// Shared memory (dynamic only, 1024-byte aligned, 128-byte swizzle everywhere):
//   Q     two [128 rows][64 dims] blocks (K-major A operand)                32 KiB
//   K     kKStages (3) stages x 16 row groups of 8 tokens: [group][half of D][8][64]    96 KiB
//   V     kVStages (3) stages, the same layout                                          96 KiB
//   xch   row maxima (and at a unit's end the sums) of both groups, per tile parity  2 KiB
// In a stage the 8-token groups sit 2048 bytes apart, the second half of D at +1024:
// Q.K^T reads K as the K-major B operand (SBO 2048), P.V reads V as the MN-major B
// operand (LBO 1024, SBO 2048).
// Tensor memory: S/P 0, 1, 2 (128 columns each) and O (128 columns).
// Pages past the unit's tokens load out of bounds and are zero-filled.
//
// Softmax (base 2): a running max is raised only when a tile's max exceeds it by more
// than 8; smaller increases are absorbed in p <= 2^8, so O is rescaled rarely.  Each
// score costs one FFMA and one ex2.approx; the sums are kept in fp32.
// Every wait is bounded; on timeout the CTA records GB_ERR_TIMEOUT, every role stops
// issuing, waits (bounded) for its own outstanding copies and MMAs, the tensor memory is
// freed and the CTA leaves.
#include <cuda.h>

#include "decode_mma.cuh"
#include "internal.cuh"
#include "ptx.cuh"
#include "tc.cuh"

namespace gb {
namespace {

constexpr int kRows = 128;     // query rows per tile (MMA M)
constexpr int kTok = 128;      // tokens per K/V tile (MMA N of Q.K^T)
constexpr int kHalf = 64;      // tokens per softmax group (MMA K of one P.V)
#ifndef GB_GROUPED_KSTAGES
#define GB_GROUPED_KSTAGES 3  // K ring depth (a K slot is free once S has read it)
#endif
#ifndef GB_GROUPED_VSTAGES
#define GB_GROUPED_VSTAGES 3  // V ring depth (a V slot is held through the softmax and P.V)
#endif
constexpr int kKStages = GB_GROUPED_KSTAGES, kVStages = GB_GROUPED_VSTAGES;
constexpr int kThreads = 352;
constexpr int kProducerWarp = 8;     // K producer, unit scheduling, Q gather
constexpr int kMmaWarp = 9;
constexpr int kVProducerWarp = 10;
constexpr int kSBufs = 3;            // S/P tiles in tensor memory
constexpr uint32_t kTmemCols = 512;  // S/P 0, 1, 2: [0, 384) (128 columns each), O: [384, 512)
constexpr uint32_t kTmemO = 384;

constexpr int kQ = 0;                // 32 KiB
constexpr int kHalfStage = 32768;    // K (or V) of one 128-token tile of one head
constexpr int kKRing = 32768;        // kKStages x 32 KiB
constexpr int kVRing = kKRing + kKStages * kHalfStage;
constexpr int kBar = kVRing + kVStages * kHalfStage;  // mbarriers and control words
constexpr int kXch = kBar + 512;     // float [2 tile parities][2 groups][128 rows]
constexpr int kSmem = kXch + 2048;

// Control area (8-byte mbarriers, then words).
constexpr int kBarKFull = 0;         // [kKStages]
constexpr int kBarKEmpty = kBarKFull + 8 * kKStages;
constexpr int kBarVFull = kBarKEmpty + 8 * kKStages;  // [kVStages]
constexpr int kBarVEmpty = kBarVFull + 8 * kVStages;
constexpr int kBarQFull = kBarVEmpty + 8 * kVStages;
constexpr int kBarQEmpty = kBarQFull + 8;
constexpr int kBarSFull = kBarQEmpty + 8;            // [kSBufs]
constexpr int kBarPFull = kBarSFull + 8 * kSBufs;    // [kSBufs]
constexpr int kBarPvDone = kBarPFull + 8 * kSBufs;   // [kSBufs]
constexpr int kBarMaxFull = kBarPvDone + 8 * kSBufs; // [2]: the two groups' row maxima of a tile are in
constexpr int kBarXchFull = kBarMaxFull + 16;
constexpr int kBarOFree = kBarXchFull + 8;
constexpr int kSchedSlots = 4;
constexpr int kBarSchedFull = kBarOFree + 8;                  // [kSchedSlots]
constexpr int kBarSchedEmpty = kBarSchedFull + 8 * kSchedSlots;  // [kSchedSlots]
constexpr int kSchedConsumers = 11;  // MMA S side, MMA P.V side, 8 softmax warps, V producer
constexpr int kWordSched = kBarSchedEmpty + 8 * kSchedSlots;  // int [kSchedSlots]: unit id, -1 = no more
constexpr int kWordTmem = kWordSched + 4 * kSchedSlots;
constexpr int kWordAbort = kWordTmem + 4;
static_assert(kWordAbort + 4 <= 512, "control area");
static_assert(kSmem <= 232448, "shared memory per block");

// K (kv = 0) or V (kv = 1) of one page of one head by 5D TMA: coordinates {0, 0, 0, kv, w},
// w = first K row / 8.
__device__ __forceinline__ void tma_page(uint32_t dst, const CUtensorMap* tm, int kv, int w, uint32_t bar) {
  asm volatile(
      "cp.async.bulk.tensor.5d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3, %4, %5, %6}], [%7];" ::"r"(
          dst),
      "l"(tm), "r"(0), "r"(0), "r"(0), "r"(kv), "r"(w), "r"(bar)
      : "memory");
}
// The same with an L2 eviction policy (a page no other query tile of its segment reads again).
__device__ __forceinline__ void tma_page_hint(uint32_t dst, const CUtensorMap* tm, int kv, int w, uint32_t bar,
                                              uint64_t pol) {
  asm volatile(
      "cp.async.bulk.tensor.5d.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint"
      " [%0], [%1, {%2, %3, %4, %5, %6}], [%7], %8;" ::"r"(dst),
      "l"(tm), "r"(0), "r"(0), "r"(0), "r"(kv), "r"(w), "r"(bar), "l"(pol)
      : "memory");
}

// Everything a role needs to know about one unit of work.
struct Unit {
  int h, s, t, sp, tok_base, Ts, ntok, seg_i0, rep, g, moff;
};

__device__ __forceinline__ Unit load_unit(const PoolView& v, long long u) {
  Unit x;
  const int tq = (int)(u / v.Hkv);
  x.h = (int)(u % v.Hkv);
  x.s = v.seg_tile_seg[tq];
  x.t = v.seg_tile_t[tq];
  x.sp = v.seg_tile_split[tq];
  const int split = v.ctl[kCtlSegSplit];
  x.tok_base = x.sp * split;
  x.Ts = min(v.seg_len[x.s] * v.P - x.tok_base, split);
  x.ntok = (x.Ts + kTok - 1) / kTok;
  x.seg_i0 = v.seg_i0[x.s];
  x.rep = v.seg_rep[x.s];
  x.g = v.seg_g[x.s];
  x.moff = v.seg_mem_off[x.s];
  return x;
}

// The grouped role of the attention kernel (k_attention, below): this CTA is one of the `ng`
// CTAs that take grouped work units; threads past kThreads only take part in the CTA's
// barriers.
template <int G>
__device__ __forceinline__ void grouped_body(const PoolView& v, const CUtensorMap* tm_p, int layer,
                                             const __nv_bfloat16* __restrict__ q, float qscale, int w_oob, int ng) {
  extern __shared__ __align__(1024) unsigned char sm[];
  const long long units = (long long)v.ctl[kCtlSegTiles] * v.Hkv;
  if (units == 0) return;
  if (smem_addr(sm) & 1023) {  // the swizzled layouts need a 1024-byte aligned base
    if (threadIdx.x == 0) set_status(v.ctl, GB_ERR_UNSUPPORTED);
    return;
  }
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const uint32_t sbase = smem_addr(sm);
  const uint32_t ctl = sbase + kBar;
  volatile int* abort_flag = reinterpret_cast<volatile int*>(sm + kBar + kWordAbort);
  if (tid == 0) {
    for (int i = 0; i < kKStages; ++i) {
      mbar_init(ctl + kBarKFull + 8 * i, 1);
      mbar_init(ctl + kBarKEmpty + 8 * i, 1);
    }
    for (int i = 0; i < kVStages; ++i) {
      mbar_init(ctl + kBarVFull + 8 * i, 1);
      mbar_init(ctl + kBarVEmpty + 8 * i, 1);
    }
    mbar_init(ctl + kBarQFull, 1);
    mbar_init(ctl + kBarQEmpty, 1);
    for (int i = 0; i < kSBufs; ++i) {
      mbar_init(ctl + kBarSFull + 8 * i, 1);
      mbar_init(ctl + kBarPFull + 8 * i, 8);
      mbar_init(ctl + kBarPvDone + 8 * i, 1);
    }
    for (int i = 0; i < 2; ++i) mbar_init(ctl + kBarMaxFull + 8 * i, 8);
    mbar_init(ctl + kBarXchFull, 8);
    mbar_init(ctl + kBarOFree, 8);
    for (int i = 0; i < kSchedSlots; ++i) {
      mbar_init(ctl + kBarSchedFull + 8 * i, 1);
      mbar_init(ctl + kBarSchedEmpty + 8 * i, kSchedConsumers);
    }
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == kMmaWarp) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(ctl + kWordTmem),
                 "r"(kTmemCols));
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *reinterpret_cast<volatile uint32_t*>(sm + kBar + kWordTmem);
  volatile int* sched = reinterpret_cast<volatile int*>(sm + kBar + kWordSched);
  constexpr int members_per_tile = kRows / G;

  if (warp == kProducerWarp) {
    // ------------------------------------------------------------------ K producer
    if (lane == 0) asm volatile("prefetch.tensormap [%0];" ::"l"(tm_p) : "memory");
    const int ppt = kTok / v.P;                     // pages per tile (2 to 16)
    const uint32_t page_bytes = (uint32_t)v.P * 256;  // K (or V) of one page of one head
    const uint64_t pol_ef = policy_evict_first();
    uint32_t n = 0;  // tiles issued
    int uidx = 0;    // units started
    bool ok = true;
    // Units come from the grid-wide counter one unit ahead: the request for the next unit
    // goes out when this one starts, so its latency hides behind this unit's tiles.  A
    // unit (or the end, -1) is published in slot uidx % kSchedSlots once every role has
    // read the unit that slot held before.
    int pending = 0;
    if (lane == 0) pending = atomicAdd(&v.ctl[kCtlGrpNext], 1);
    // The next unit's description is loaded while this unit's second tile is issued, so at
    // the unit boundary only its page ids and member rows (loaded together) are waited for.
    Unit xn{};
    bool have_xn = false;
    for (;; ++uidx) {
      if (!ok || *abort_flag) break;
      const long long u = __shfl_sync(0xffffffffu, pending, 0);
      if (lane == 0 && u < units) pending = atomicAdd(&v.ctl[kCtlGrpNext], 1);
      const int k = uidx & (kSchedSlots - 1);
      if (lane == 0 && uidx >= kSchedSlots)
        ok = wait_or_abort(ctl + kBarSchedEmpty + 8 * k, ((uidx / kSchedSlots) - 1) & 1, abort_flag);
      ok = __shfl_sync(0xffffffffu, ok ? 1 : 0, 0) != 0;
      if (!ok) break;
      if (lane == 0) {
        sched[k] = u < units ? (int)u : -1;
        mbar_arrive(ctl + kBarSchedFull + 8 * k);
      }
      if (u >= units) break;
      const Unit x = have_xn ? xn : load_unit(v, u);
      have_xn = false;
      // Query rows of the unit: row r = (member, query head of this KV head); lane l takes rows
      // l, l + 32, l + 64, l + 96.  Their member beams are loaded now, beside the first page ids.
      const char* qrow[kRows / 32];
      bool qvalid[kRows / 32];
#pragma unroll
      for (int i = 0; i < kRows / 32; ++i) {
        const int r = lane + 32 * i;
        const int m = x.t * members_per_tile + r / G, gg = r % G;
        qvalid[i] = m < x.g;
        const int b = qvalid[i] ? v.seg_members[x.moff + m] / kMaxSegDepth : 0;
        qrow[i] = reinterpret_cast<const char*>(q + ((size_t)b * v.Hq + (size_t)x.h * G + gg) * 128);
      }
      int page_l = 0;
      for (int j = 0; j < x.ntok; ++j, ++n) {
        if (j == 1) {  // prefetch the next unit's description (its id came back with this unit)
          const long long un = __shfl_sync(0xffffffffu, pending, 0);
          if (un < units) {
            xn = load_unit(v, un);
            have_xn = true;
          }
        }
        const uint32_t st = n % kKStages;
        const int pb = j * ppt;  // first page of the tile within the unit
        if ((pb & 31) == 0) {
          const int tl = (pb + lane) * v.P;
          page_l = tl < x.Ts ? v.tables[(size_t)x.rep * v.max_pages + x.seg_i0 + (x.tok_base + tl) / v.P] : 0;
        }
        // Lane c < ppt: row group of page c's K slab (pages past the unit load zeros).
        int w = w_oob;
        {
          const int page_c = __shfl_sync(0xffffffffu, page_l, (pb + (lane & 15)) & 31);
          const int tl = j * kTok + lane * v.P;  // token within the unit
          if (lane < ppt && tl < x.Ts) {
            int page = page_c;
            if (page < 0 || page >= v.num_pages) {
              set_status(v.ctl, GB_ERR_INVALID);
              page = 0;
            }
            const long long slab = (((long long)layer * v.num_pages + page) * 2) * v.Hkv + x.h;
            w = (int)(slab * v.P / 8);
          }
        }
        if (lane == 0 && n >= (uint32_t)kKStages)
          ok = wait_or_abort(ctl + kBarKEmpty + 8 * st, ((n / kKStages) - 1) & 1, abort_flag);
        ok = __shfl_sync(0xffffffffu, ok ? 1 : 0, 0) != 0;
        if (!ok) break;
        const uint32_t bar = ctl + kBarKFull + 8 * st;
        if (lane == 0) mbar_arrive_expect_tx(bar, kHalfStage);
        __syncwarp();
        // Lane c issues page c: a TMA instruction holds its thread for a while, so the
        // lanes' copies go out in parallel.
        if (lane < ppt) {
          // The segment's only query tile reads its pages once: evict them first, before data
          // that is read again (the queries, the records, other tiles' pages).
          if (x.g * G <= kRows)
            tma_page_hint(sbase + kKRing + st * kHalfStage + lane * page_bytes, tm_p, 0, w, bar, pol_ef);
          else
            tma_page(sbase + kKRing + st * kHalfStage + lane * page_bytes, tm_p, 0, w, bar);
        }
        if (j == 0) {
          // Query rows of the unit (after its first tile's copies are under way): row r =
          // (member, query head of this KV head); zero rows past the members.  The single
          // Q buffer is free once the previous unit's last S has completed.
          if (lane == 0 && uidx >= 1) ok = wait_or_abort(ctl + kBarQEmpty, (uidx - 1) & 1, abort_flag);
          ok = __shfl_sync(0xffffffffu, ok ? 1 : 0, 0) != 0;
          if (!ok) {
            ++n;
            break;
          }
          // All 64 16-byte pieces of the lane's rows go out as asynchronous copies into the
          // swizzled layout, so the whole 32 KiB is in flight at once; rows past the members
          // are zeroed.  Query rows are read by every unit of their beams: keep them in L2 against the
          // stream of K/V tiles (evict-last).
          const uint64_t qpol = policy_evict_last();
#pragma unroll
          for (int i = 0; i < kRows / 32; ++i)
#pragma unroll
            for (int c = 0; c < 16; ++c) {
              const uint32_t dst = sbase + kQ + (c >> 3) * 16384 + swz(lane + 32 * i, (c & 7) * 8);
              if (qvalid[i])
                asm volatile("cp.async.cg.shared.global.L2::cache_hint [%0], [%1], 16, %2;" ::"r"(dst),
                             "l"(qrow[i] + 16 * c), "l"(qpol)
                             : "memory");
              else
                *reinterpret_cast<uint4*>(sm + (dst - sbase)) = make_uint4(0, 0, 0, 0);
            }
          asm volatile("cp.async.commit_group;\n\tcp.async.wait_group 0;" ::: "memory");
          fence_proxy_async_smem();
          __syncwarp();
          if (lane == 0) mbar_arrive(ctl + kBarQFull);
        }
      }
    }
    // Drain: copies still in flight land before the CTA leaves (bounded).
    if (lane == 0 && *abort_flag) {
      for (uint32_t k = n > (uint32_t)kKStages ? n - kKStages : 0; k < n; ++k)
        mbar_wait_bounded(ctl + kBarKFull + 8 * (k % kKStages), (k / kKStages) & 1, kWaitLimitNs / 8);
    }
  } else if (warp == kVProducerWarp) {
    // ------------------------------------------------------------------ V producer
    const int ppt = kTok / v.P;
    const uint32_t page_bytes = (uint32_t)v.P * 256;
    const uint64_t pol_ef = policy_evict_first();
    uint32_t n = 0;  // tiles issued
    bool ok = true;
    for (int uidx = 0; ok; ++uidx) {
      const int k = uidx & (kSchedSlots - 1);
      if (lane == 0) ok = wait_or_abort(ctl + kBarSchedFull + 8 * k, (uidx / kSchedSlots) & 1, abort_flag);
      ok = __shfl_sync(0xffffffffu, ok ? 1 : 0, 0) != 0;
      if (!ok) break;
      const int id = sched[k];
      __syncwarp();
      if (lane == 0) mbar_arrive(ctl + kBarSchedEmpty + 8 * k);
      if (id < 0) break;
      const Unit x = load_unit(v, id);
      int page_l = 0;
      for (int j = 0; j < x.ntok; ++j, ++n) {
        const uint32_t st = n % kVStages;
        const int pb = j * ppt;
        if ((pb & 31) == 0) {
          const int tl = (pb + lane) * v.P;
          page_l = tl < x.Ts ? v.tables[(size_t)x.rep * v.max_pages + x.seg_i0 + (x.tok_base + tl) / v.P] : 0;
        }
        int w = w_oob;
        {
          const int page_c = __shfl_sync(0xffffffffu, page_l, (pb + (lane & 15)) & 31);
          const int tl = j * kTok + lane * v.P;
          if (lane < ppt && tl < x.Ts) {
            int page = page_c;
            if (page < 0 || page >= v.num_pages) page = 0;  // recorded by the K producer
            const long long slab = (((long long)layer * v.num_pages + page) * 2) * v.Hkv + x.h;
            w = (int)(slab * v.P / 8);
          }
        }
        if (lane == 0 && n >= (uint32_t)kVStages)
          ok = wait_or_abort(ctl + kBarVEmpty + 8 * st, ((n / kVStages) - 1) & 1, abort_flag);
        ok = __shfl_sync(0xffffffffu, ok ? 1 : 0, 0) != 0;
        if (!ok) break;
        const uint32_t bar = ctl + kBarVFull + 8 * st;
        if (lane == 0) mbar_arrive_expect_tx(bar, kHalfStage);
        __syncwarp();
        if (lane < ppt) {
          // The segment's only query tile reads its pages once: evict them first, before data
          // that is read again (the queries, the records, other tiles' pages).
          if (x.g * G <= kRows)
            tma_page_hint(sbase + kVRing + st * kHalfStage + lane * page_bytes, tm_p, 1, w, bar, pol_ef);
          else
            tma_page(sbase + kVRing + st * kHalfStage + lane * page_bytes, tm_p, 1, w, bar);
        }
      }
    }
    if (lane == 0 && *abort_flag) {
      for (uint32_t k = n > (uint32_t)kVStages ? n - kVStages : 0; k < n; ++k)
        mbar_wait_bounded(ctl + kBarVFull + 8 * (k % kVStages), (k / kVStages) & 1, kWaitLimitNs / 8);
    }
  } else if (warp == kMmaWarp) {
    // ------------------------------------------------------------------ MMA issuer
    constexpr uint32_t ID_S = idesc(kRows, kTok, false);
    constexpr uint32_t ID_PV = idesc(kRows, 128, true);
    uint32_t n_s = 0, n_pv = 0;  // S and P.V tiles issued
    bool alive = true;
    int uidx_s = 0, j_s = 0;     // the tile of the next S: unit index, tile in unit
    bool have_s = false, done_s = false;
    Unit xs{};
    // S(n_s) can go when its unit is known, the Q buffer holds that unit (first tile), its
    // stage has landed and P.V(n_s - 2), the last reader of its S/P columns, has been issued.
    auto s_ready = [&]() -> bool {
      if (!have_s) {
        const int k = uidx_s & (kSchedSlots - 1);
        if (!mbar_test(ctl + kBarSchedFull + 8 * k, (uidx_s / kSchedSlots) & 1)) return false;
        const int id = sched[k];
        mbar_arrive(ctl + kBarSchedEmpty + 8 * k);
        if (id < 0) {
          done_s = true;
          return false;
        }
        xs = load_unit(v, id);
        have_s = true;
        j_s = 0;
      }
      if (j_s == 0 && !mbar_test(ctl + kBarQFull, uidx_s & 1)) return false;
      if (!mbar_test(ctl + kBarKFull + 8 * (n_s % kKStages), (n_s / kKStages) & 1)) return false;
      return n_pv + (kSBufs - 1) >= n_s;
    };
    auto issue_s = [&]() {
      const uint32_t st = n_s % kKStages, sb = n_s % kSBufs;
      tc_fence_after();
      const uint32_t kb = sbase + kKRing + st * kHalfStage;
#pragma unroll
      for (int kk = 0; kk < 8; ++kk) {
        const uint64_t a = sdesc(sbase + kQ + (kk >> 2) * 16384 + (kk & 3) * 32, 16, 1024);
        const uint64_t b = sdesc(kb + (kk >> 2) * 1024 + (kk & 3) * 32, 16, 2048);
        mma(tmem + sb * 128, a, b, ID_S, kk > 0);
      }
      mma_commit(ctl + kBarKEmpty + 8 * st);  // the K slot is free once S has read it
      mma_commit(ctl + kBarSFull + 8 * sb);
      if (j_s + 1 == xs.ntok) mma_commit(ctl + kBarQEmpty);  // last read of the Q buffer for this unit
      ++n_s;
      if (++j_s == xs.ntok) {
        ++uidx_s;
        have_s = false;
      }
    };
    if (lane == 0) {
      int uidx_p = 0, j_p = 0;    // the tile of the next P.V
      bool have_p = false;
      Unit xp{};
      uint64_t t_progress = globaltimer_ns();
      uint32_t spins = 0;
      for (;;) {
        bool progressed = false;
        if (!done_s && s_ready()) {
          issue_s();
          progressed = true;
        }
        if (!have_p) {
          const int k = uidx_p & (kSchedSlots - 1);
          if (mbar_test(ctl + kBarSchedFull + 8 * k, (uidx_p / kSchedSlots) & 1)) {
            const int id = sched[k];
            mbar_arrive(ctl + kBarSchedEmpty + 8 * k);
            if (id < 0) break;  // every unit's P.V has been issued
            xp = load_unit(v, id);
            have_p = true;
            j_p = 0;
            progressed = true;
          }
        }
        const uint32_t pb = n_pv % kSBufs, st = n_pv % kVStages;
        // P.V(n) needs both groups' P; a unit's first P.V also needs the previous unit's
        // accumulator read out (o_free), since it overwrites it.
        if (have_p && n_pv < n_s && mbar_test(ctl + kBarPFull + 8 * pb, (n_pv / kSBufs) & 1) &&
            mbar_test(ctl + kBarVFull + 8 * st, (n_pv / kVStages) & 1) &&
            (j_p > 0 || uidx_p == 0 || mbar_test(ctl + kBarOFree, (uidx_p - 1) & 1))) {
          tc_fence_after();
          const uint32_t vb = sbase + kVRing + st * kHalfStage;
#pragma unroll
          for (int k = 0; k < 2; ++k)
#pragma unroll
            for (int kk = 0; kk < kHalf / 16; ++kk) {
              // A = P_k (bf16 pairs, 8 columns per 16 tokens), B = V tokens [64k + 16kk, +16).
              const uint64_t b = sdesc(vb + (k * 4 + kk) * 4096, 1024, 2048);
              mma_ts(tmem + kTmemO, tmem + pb * 128 + k * 64 + kk * 8, b, ID_PV,
                     (j_p > 0 || k > 0 || kk > 0) ? 1u : 0u);
            }
          mma_commit(ctl + kBarVEmpty + 8 * st);
          mma_commit(ctl + kBarPvDone + 8 * pb);
          ++n_pv;
          if (++j_p == xp.ntok) {
            ++uidx_p;
            have_p = false;
          }
          progressed = true;
        }
        if (progressed) {
          spins = 0;
        } else if ((++spins & 255) == 0) {
          const uint64_t now = globaltimer_ns();
          if (spins == 256) t_progress = now;  // first check after the last progress
          if (*abort_flag || now - t_progress > kWaitLimitNs) {
            *abort_flag = 1;
            alive = false;
            break;
          }
        }
      }
      if (!alive) {
        // Let issued MMAs finish before the tensor memory is freed (bounded).
        if (n_pv > 0)
          mbar_wait_bounded(ctl + kBarPvDone + 8 * ((n_pv - 1) % kSBufs), ((n_pv - 1) / kSBufs) & 1, kWaitLimitNs / 8);
        if (n_s > 0)
          mbar_wait_bounded(ctl + kBarSFull + 8 * ((n_s - 1) % kSBufs), ((n_s - 1) / kSBufs) & 1, kWaitLimitNs / 8);
      }
    }
    __syncwarp();
  } else if (warp > kVProducerWarp) {
    // threads past the grouped role's kThreads (the attention kernel's block holds the
    // per-beam role's 12 warps): nothing to do but the CTA's barriers
  } else {
    // ------------------------------------------------------------------ softmax (warps 0-7)
    // Both groups keep the same running max per row (they swap their tile maxima through
    // shared memory), so their P.V products add into one accumulator O.
    const int grp = warp >> 2;           // softmax group: tokens [64 grp, 64 grp + 64) of each tile
    const int r = tid & 127;             // query row / TMEM lane
    const uint32_t lane_base = (uint32_t)((warp & 3) * 32) << 16;
    const uint32_t o_half = tmem + kTmemO + grp * 64 + lane_base;  // this group's half of O's columns
    float* xch = reinterpret_cast<float*>(sm + kXch);  // [tile parity][group][row]
    uint32_t n = 0;
    int uidx = 0;
    bool alive = true;
    for (;; ++uidx) {
      const int k = uidx & (kSchedSlots - 1);
      if (!wait_or_abort(ctl + kBarSchedFull + 8 * k, (uidx / kSchedSlots) & 1, abort_flag)) break;
      const int id = sched[k];
      __syncwarp();
      if (lane == 0) mbar_arrive(ctl + kBarSchedEmpty + 8 * k);
      if (id < 0) break;
      const Unit x = load_unit(v, id);
      // This row's record (member beam, its record slot): loaded now, used at the unit's
      // end, so the two dependent loads complete behind the unit's tiles.
      const int m = x.t * members_per_tile + r / G, gg = r % G;
      const int bk = m < x.g ? v.seg_members[x.moff + m] : 0;
      const int r_idx = v.seg_rec_off[bk] + x.sp;
      float m_ref = -INFINITY, l = 0.f;
      for (int j = 0; j < x.ntok; ++j, ++n) {
        const uint32_t sb = n % kSBufs;
        const uint32_t sp_addr = tmem + sb * 128 + grp * 64 + lane_base;
        if (!wait_or_abort(ctl + kBarSFull + 8 * sb, (n / kSBufs) & 1, abort_flag)) { alive = false; break; }
        tc_fence_after();
        const int valid = min(max(x.Ts - j * kTok - grp * kHalf, 0), kHalf);  // this group's tokens in the tile
        float sv[kHalf];
        float mt_own = -INFINITY;
        if (valid > 0) {
          tmem_ld32(sp_addr, sv);
          tmem_ld32(sp_addr + 32, sv + 32);
          if (valid < kHalf) {  // only a unit's last tile reaches past its tokens
#pragma unroll
            for (int c = 0; c < kHalf; ++c)
              if (c >= valid) sv[c] = -INFINITY;
          }
          // Max on the raw scores; qscale > 0, so it scales to the max in log2 units.
          float mr0 = sv[0], mr1 = sv[1], mr2 = sv[2], mr3 = sv[3];
#pragma unroll
          for (int c = 4; c < kHalf; c += 4) {
            mr0 = fmaxf(mr0, sv[c]);
            mr1 = fmaxf(mr1, sv[c + 1]);
            mr2 = fmaxf(mr2, sv[c + 2]);
            mr3 = fmaxf(mr3, sv[c + 3]);
          }
          mt_own = fmaxf(fmaxf(mr0, mr1), fmaxf(mr2, mr3)) * qscale;
        }
        // The tile's row max over both groups: slot n & 1 is rewritten two tiles later,
        // after every warp has passed this tile's barrier, so after it has been read.
        const int slot = n & 1;
        xch[(slot * 2 + grp) * 128 + r] = mt_own;
        __syncwarp();
        if (lane == 0) mbar_arrive(ctl + kBarMaxFull + 8 * slot);
        if (!wait_or_abort(ctl + kBarMaxFull + 8 * slot, (n >> 1) & 1, abort_flag)) { alive = false; break; }
        const float mt = fmaxf(mt_own, xch[(slot * 2 + 1 - grp) * 128 + r]);
        const bool raise = mt > m_ref + 8.f;
        if (j > 0 && __any_sync(0xffffffffu, raise)) {
          // O must hold P.V(n-1) and nothing newer before it is rescaled; each group
          // rescales its half of the columns.
          if (!wait_or_abort(ctl + kBarPvDone + 8 * ((n - 1) % kSBufs), ((n - 1) / kSBufs) & 1, abort_flag)) {
            alive = false;
            break;
          }
          tc_fence_after();
          const float alpha = raise ? exp2f(m_ref - mt) : 1.f;
#pragma unroll 1
          for (int c0 = 0; c0 < 64; c0 += 32) {
            float o[32];
            tmem_ld32(o_half + c0, o);
#pragma unroll
            for (int i = 0; i < 32; ++i) o[i] *= alpha;
            tmem_st32(o_half + c0, o);
          }
          if (raise) l *= alpha;
        }
        if (raise) m_ref = mt;
        uint32_t pw[kHalf / 2];
        if (valid == 0) {
#pragma unroll
          for (int i = 0; i < kHalf / 2; ++i) pw[i] = 0u;
        } else {
          const float neg_m = -m_ref;
          float l0 = 0.f, l1 = 0.f, l2 = 0.f, l3 = 0.f;
#pragma unroll
          for (int c = 0; c < kHalf; c += 4) {
            // p = 2^(s * qscale - m); masked scores give 2^-inf = 0.
            const float p0 = ex2_approx(fmaf(sv[c], qscale, neg_m));
            const float p1 = ex2_approx(fmaf(sv[c + 1], qscale, neg_m));
            const float p2 = ex2_approx(fmaf(sv[c + 2], qscale, neg_m));
            const float p3 = ex2_approx(fmaf(sv[c + 3], qscale, neg_m));
            const __nv_bfloat162 pr0 = __floats2bfloat162_rn(p0, p1);
            const __nv_bfloat162 pr1 = __floats2bfloat162_rn(p2, p3);
            pw[c / 2] = *reinterpret_cast<const uint32_t*>(&pr0);
            pw[c / 2 + 1] = *reinterpret_cast<const uint32_t*>(&pr1);
            l0 += p0;
            l1 += p1;
            l2 += p2;
            l3 += p3;
          }
          l += (l0 + l1) + (l2 + l3);
        }
        tmem_st32u(sp_addr, pw);  // P_k over the first 32 of this group's S columns
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(ctl + kBarPFull + 8 * sb);
      }
      if (!alive) break;
      // Unit end: O is final once P.V of the last tile has completed.  The groups add their
      // row sums (same max); slot n & 1 is free (its last reader passed the previous tile).
      const uint32_t last = n - 1;
      if (!wait_or_abort(ctl + kBarPvDone + 8 * (last % kSBufs), (last / kSBufs) & 1, abort_flag)) break;
      tc_fence_after();
      const int slot = n & 1;
      xch[(slot * 2 + grp) * 128 + r] = l;
      __syncwarp();
      if (lane == 0) mbar_arrive(ctl + kBarXchFull);
      if (!wait_or_abort(ctl + kBarXchFull, uidx & 1, abort_flag)) break;
      const float l_all = l + xch[(slot * 2 + 1 - grp) * 128 + r];
      const int b = bk / kMaxSegDepth;
      const bool has = m < x.g && r_idx < kMaxSegRecords;
      float* rec = v.grec + (((size_t)b * kMaxSegRecords + r_idx) * v.Hkv + x.h) * v.record_floats;
      const uint64_t rpol = policy_evict_last();  // the merge reads the record back from L2
      // Group k writes columns [64k, 64k + 64) of the output.
#pragma unroll 1
      for (int c0 = 0; c0 < 64; c0 += 32) {  // warp-collective loads: every lane takes part
        float o[32];
        tmem_ld32(o_half + c0, o);
        if (has) {
#pragma unroll
          for (int i = 0; i < 32; i += 4)
            st_hint4(rec + gg * 128 + grp * 64 + c0 + i, make_float4(o[i], o[i + 1], o[i + 2], o[i + 3]), rpol);
        }
      }
      if (has && grp == 0) {
        st_hint(rec + G * 128 + gg, m_ref, rpol);
        st_hint(rec + G * 128 + G + gg, l_all, rpol);
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(ctl + kBarOFree);
      // Every warp has read this unit's sums before the next unit's first tile rewrites
      // the exchange slot.
      if (!wait_or_abort(ctl + kBarOFree, uidx & 1, abort_flag)) break;
    }
  }

  if (*abort_flag && tid == 0) set_status(v.ctl, GB_ERR_TIMEOUT);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == kMmaWarp) asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kTmemCols));
  // Every copy and MMA has completed: the barriers' memory may serve the per-beam role next.
  if (tid == 0)
    for (int b = 0; b < kWordSched; b += 8) mbar_inval(ctl + b);
}

constexpr int kAttnThreads = kMmaWarps * 32;  // the per-beam role's 12 warps; the grouped role uses 11
static_assert(kAttnThreads >= kThreads, "the grouped role's warps fit the block");
constexpr int kAttnSmem = kSmem > DecodeMmaSmem::TOTAL ? kSmem : DecodeMmaSmem::TOTAL;

// The attention phase of a step with shared-prefix segments, in one launch: the grouped role
// (the tcgen05 kernel above) and the per-beam role (the warp-MMA kernel of decode_mma.cuh)
// over the step's unshared tails, one CTA per SM at a time.  When the step reads little per SM
// (decode_ctas), both roles are latency-bound and run side by side, each on its share of the
// SMs; otherwise the per-beam CTAs follow the grouped ones onto the SMs they leave.  The
// pairs' records are merged into `out` in the same launch (combine.cuh).
template <int G>
__global__ void __launch_bounds__(kAttnThreads, 1)
    k_attention(PoolView v, const __grid_constant__ CUtensorMap tmg, const __grid_constant__ CUtensorMap tmd,
                const __grid_constant__ CUtensorMap tmdh, int layer, const __nv_bfloat16* __restrict__ q,
                float qscale, int w_oob, float* __restrict__ out) {
  pdl_wait();
  pdl_launch_dependents();
  // Grid of 2 S CTAs (S = SM count).  Large steps: CTAs [0, S) take the grouped role and
  // leave, CTAs [S, 2S) the per-beam role, each on an SM as a grouped CTA leaves it (CTAs
  // start in index order), and merge the records; a grouped CTA never waits, so every
  // per-beam CTA gets an SM.  Small steps: [0, ng) grouped and [ng, S) per-beam side by side,
  // all S resident at once, all S merging; the rest leave at once.
  const int S = (int)gridDim.x / 2, c = (int)blockIdx.x;
  const bool ok = v.ctl[kCtlStepOk] != 0;
  int nd = S, ng = S;
  if (ok) {
    nd = decode_ctas(v, S);
    if (nd < S) ng = S - nd;
  }
  const bool split = nd < S;
  const int pb0 = split ? ng : S;  // first per-beam CTA
  if (c >= pb0 + nd) return;
  if (c < pb0) {
    if (ok) {
      grouped_body<G>(v, &tmg, layer, q, qscale, w_oob, ng);
      grouped_cta_done(v);
    }
    if (!split) return;
  } else {
    decode_mma_body<G>(v, &tmd, &tmdh, layer, q, qscale, 1, c - pb0, nd);
  }
  // A large step's per-beam CTAs start as grouped CTAs leave, so they take the pairs as they
  // finish; a small step's CTAs all start together and split the pairs evenly.
  if (split) combine_pairs<G>(v, 1, nd * kMmaWarps, ng, false, c, S, out);
  else combine_pairs<G>(v, 1, nd * kMmaWarps, ng, true, c - S, S, out);
}

}  // namespace

// 5D tensor maps over the whole pool, which is viewed as rows of D = 128 bf16 (256 bytes):
// dims {64 dims, 8 rows, 2 halves of D, K|V, row groups of 8}, strides {256, 128,
// Hkv * P * 256 (K slab to V slab), 2048} bytes.  The grouped kernel's box {64, 8, 2, 1,
// P / 8} is K (K|V coordinate 0) or V (coordinate 1) of one page of one head; the per-beam
// kernel's box {64, 8, 2, 2, 2} is K and V of 16 tokens of one head.  A box lands in shared
// memory in the dims' order ([row group][K|V][half][8 rows][64 dims]) with the 128-byte
// swizzle.  The row-group extent ends with the last K slab, so every coordinate in range
// addresses a real K and V slab.  Sets have_tmap (grouped) and have_dtmap (per-beam).
void make_kv_tensor_maps(gb_pool* pool) {
  typedef CUresult (*EncodeFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                               const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                               CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);
  static EncodeFn encode = nullptr;
  pool->have_tmap = pool->have_dtmap = false;
  if (!encode) {
    cudaDriverEntryPointQueryResult qr;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", reinterpret_cast<void**>(&encode), 12000,
                                         cudaEnableDefault, &qr) != cudaSuccess ||
        qr != cudaDriverEntryPointSuccess || !encode)
      return;
  }
  const PoolView& v = pool->view;
  if (v.dtype != GB_BF16 || v.D != 128) return;
  const unsigned long long rows = (unsigned long long)v.layers * v.num_pages * 2 * v.Hkv * v.P;
  if (rows >= (1ull << 31)) return;
  cuuint64_t dims[5] = {64, 8, 2, 2, (rows - (unsigned long long)v.Hkv * v.P) / 8};
  cuuint64_t strides[4] = {256, 128, (cuuint64_t)v.Hkv * v.P * 256, 2048};
  cuuint32_t es[5] = {1, 1, 1, 1, 1};
  pool->tmap_oob = (int)dims[4];
  if (v.P % 8 == 0 && kTok % v.P == 0 && kTok / v.P <= 16) {
    cuuint32_t box[5] = {64, 8, 2, 1, (cuuint32_t)(v.P / 8)};
    pool->have_tmap = encode(reinterpret_cast<CUtensorMap*>(pool->tmap), CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 5, v.kv,
                             dims, strides, box, es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                             CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
  }
  if (v.P % 16 == 0) {
    cuuint32_t box[5] = {64, 8, 2, 2, 2};
    cuuint32_t half[5] = {64, 8, 2, 2, 1};  // the first 8 tokens of a chunk only
    pool->have_dtmap = encode(reinterpret_cast<CUtensorMap*>(pool->dtmap), CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 5, v.kv,
                              dims, strides, box, es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                              CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS &&
                       encode(reinterpret_cast<CUtensorMap*>(pool->dtmap_half), CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 5,
                              v.kv, dims, strides, half, es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                              CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
  }
}

template <int G>
static cudaError_t launch_attention_t(gb_pool* pool, int layer, const void* q, float scale, float* out,
                                      cudaStream_t s) {
  {
    const cudaError_t e = set_max_dynamic_smem(reinterpret_cast<const void*>(k_attention<G>), kAttnSmem);
    if (e != cudaSuccess) return e;
  }
  const PoolView& v = pool->view;
  const float qscale = scale * 1.4426950408889634f;
  prof_begin(pool, GB_PROF_GROUPED, s);
  prof_begin(pool, GB_PROF_DECODE, s);
  const cudaError_t e = launch_pdl(k_attention<G>, 2 * pool->num_sms, kAttnThreads, kAttnSmem, s, v,
                                   *reinterpret_cast<const CUtensorMap*>(pool->tmap),
                                   *reinterpret_cast<const CUtensorMap*>(pool->dtmap),
                                   *reinterpret_cast<const CUtensorMap*>(pool->dtmap_half), layer,
                                   static_cast<const __nv_bfloat16*>(q), qscale, pool->tmap_oob, out);
  prof_end(pool, GB_PROF_DECODE, s);
  prof_end(pool, GB_PROF_GROUPED, s);
  pool->launches += 1;
  return e;
}

cudaError_t launch_attention(gb_pool* pool, int layer, const void* q, float scale, float* out, cudaStream_t s) {
  switch (pool->view.G) {
    case 2: return launch_attention_t<2>(pool, layer, q, scale, out, s);
    case 4: return launch_attention_t<4>(pool, layer, q, scale, out, s);
    case 8: return launch_attention_t<8>(pool, layer, q, scale, out, s);
  }
  return cudaErrorInvalidValue;
}

}  // namespace gb
