// Shared-prefix segments for the grouped attention path.
//
// A branched child shares every full page of its parent's prefix (Section 3.1,
// after Eq. 3), so the beams that hold the page at table index i are exactly the
// beams that also share every index before i.  Along one beam's table the number
// of sharers (the page refcount) therefore never increases, and it changes exactly
// where the set of sharers changes.  A segment is a maximal run of full pages of one
// beam with a constant sharer set of at least `group_min` beams; every sharer of a
// segment sees the same run at the same table indices.  The grouped kernel reads a
// segment's pages once for all its sharers instead of once per beam.
//
// Rebuild (after seed, prune/branch and release; the set only changes there):
//   1. scan:    one warp per beam walks its table, records the starts of its
//               segments (up to kMaxSegDepth) and how many leading pages they cover,
//               and marks each start page with the lowest beam that starts there;
//   2. lead:    the lowest beam of each segment creates it (id, pages, member count);
//   3. members: every member appends (beam, depth) to its segment's member list;
//   4. tiles:   one CTA lays the segments' 128-row query tiles out as a flat list.
// Segment ids and member order follow atomics, but each output row is computed
// independently of its position, so results do not depend on that order.
#include "internal.cuh"

namespace gb {

constexpr int kSegLenBuckets = 256;  // work-list entries sorted by length in 128-token tiles (longer ones share the last bucket)

__global__ void k_seg_scan(PoolView v, unsigned long long gen) {
  pdl_wait();
  pdl_launch_dependents();
  const int lane = threadIdx.x & 31;
  const int b = (int)((blockIdx.x * (long long)blockDim.x + threadIdx.x) >> 5);
  if (blockIdx.x == 0 && threadIdx.x == 0) {
    v.ctl[kCtlSegCount] = 0;
    v.ctl[kCtlSegMembers] = 0;
    v.ctl[kCtlSegTiles] = 0;
  }
  if (b >= v.max_beams) return;
  int cover = 0, nseg = 0;
  if (v.grouped && v.active[b]) {
    const int nfull = v.seq_len[b] / v.P;
    const int* tb = v.tables + (size_t)b * v.max_pages;
    int prev_g = -1;
    for (int i0 = 0; i0 < nfull; i0 += 32) {
      const int i = i0 + lane;
      int p = -1, g = 0;
      if (i < nfull) {
        p = tb[i];
        g = (p >= 0 && p < v.num_pages) ? v.refcnt[p] : 0;
      }
      const unsigned low = __ballot_sync(0xffffffffu, i < nfull && g < v.group_min);
      const int valid = min(32, nfull - i0);
      const int lim = low ? min(valid, __ffs(low) - 1) : valid;  // positions still covered in this chunk
      int gprev = __shfl_up_sync(0xffffffffu, g, 1);
      if (lane == 0) gprev = prev_g;
      unsigned starts = __ballot_sync(0xffffffffu, lane < lim && g != gprev);
      bool stop = low != 0 || lim < 32;
      while (starts) {
        const int l = __ffs(starts) - 1;
        starts &= starts - 1;
        if (nseg == kMaxSegDepth) {  // deeper levels stay on the per-beam path
          cover = i0 + l;
          stop = true;
          goto done;
        }
        const int pl = __shfl_sync(0xffffffffu, p, l);
        if (lane == 0) {
          v.seg_bstart[b * kMaxSegDepth + nseg] = i0 + l;
          v.seg_bpage[b * kMaxSegDepth + nseg] = pl;
          atomicMax(&v.seg_owner[pl], (gen << 32) | (unsigned long long)(0xffffffffu - (unsigned)b));
        }
        ++nseg;
      }
      cover = i0 + lim;
      if (stop) break;
      prev_g = __shfl_sync(0xffffffffu, g, 31);
    }
  }
done:
  if (lane == 0) {
    v.seg_cover[b] = cover;
    v.seg_nseg[b] = nseg;
  }
}

__global__ void k_seg_lead(PoolView v, unsigned long long gen) {
  pdl_wait();
  pdl_launch_dependents();
  const int idx = blockIdx.x * blockDim.x + threadIdx.x;
  const int b = idx / kMaxSegDepth, k = idx % kMaxSegDepth;
  if (b >= v.max_beams || k >= v.seg_nseg[b]) return;
  const int p0 = v.seg_bpage[b * kMaxSegDepth + k];
  const unsigned long long ow = v.seg_owner[p0];
  if ((ow >> 32) != gen || (0xffffffffu - (unsigned)(ow & 0xffffffffu)) != (unsigned)b) return;
  const int id = atomicAdd(&v.ctl[kCtlSegCount], 1);
  const int g = v.refcnt[p0];
  const int off = atomicAdd(&v.ctl[kCtlSegMembers], g);
  const int i0 = v.seg_bstart[b * kMaxSegDepth + k];
  const int end = (k + 1 < v.seg_nseg[b]) ? v.seg_bstart[b * kMaxSegDepth + k + 1] : v.seg_cover[b];
  v.seg_i0[id] = i0;
  v.seg_len[id] = end - i0;
  v.seg_rep[id] = b;
  v.seg_g[id] = g;
  v.seg_mem_off[id] = off;
  v.seg_fill[id] = 0;
  v.seg_id[p0] = id;
}

__global__ void k_seg_members(PoolView v) {
  pdl_wait();
  pdl_launch_dependents();
  const int idx = blockIdx.x * blockDim.x + threadIdx.x;
  const int b = idx / kMaxSegDepth, k = idx % kMaxSegDepth;
  if (b >= v.max_beams || k >= v.seg_nseg[b]) return;
  const int id = v.seg_id[v.seg_bpage[b * kMaxSegDepth + k]];
  v.seg_bid[idx] = id;
  const int slot = atomicAdd(&v.seg_fill[id], 1);
  const int cap = v.max_beams * kMaxSegDepth;
  if (slot < v.seg_g[id] && v.seg_mem_off[id] + slot < cap) v.seg_members[v.seg_mem_off[id] + slot] = idx;
}

#ifndef GB_SEG_UNITS_PCT
#define GB_SEG_UNITS_PCT 200  // grouped work units aimed at per multiprocessor, in percent
#endif

// One CTA: the grouped work list.  Each segment has ceil(g*G/128) query tiles; each
// tile is split along the segment's tokens into pieces of `split` tokens (a multiple of
// the grouped kernel's 128-token K/V tile) so that the list has about two units per
// multiprocessor (and no beam needs more than
// kMaxSegRecords partial records).  Entries are (segment, tile, split); every beam
// gets the offsets of its records (one per split of each of its segments).
__global__ void __launch_bounds__(1024) k_seg_tiles(PoolView v) {
  pdl_wait();
  pdl_launch_dependents();
  __shared__ int tmp[33];
  __shared__ int s_split, s_total;
  __shared__ int hist[kSegLenBuckets];
  const int nseg = v.ctl[kCtlSegCount];
  const int rows_per_tile = 128;
  const int cap = v.max_beams * kMaxSegRecords;
  int rowtok = 0, tiletok = 0, segtok = 0;
  for (int base = 0; base < nseg; base += blockDim.x) {
    const int s = base + threadIdx.x;
    const int tiles = s < nseg ? (v.seg_g[s] * v.G + rows_per_tile - 1) / rows_per_tile : 0;
    const int toks = s < nseg ? v.seg_len[s] * v.P : 0;
    int t1, t2, t3;
    block_exclusive_scan(s < nseg ? v.seg_g[s] * v.G * toks : 0, tmp, &t1);
    block_exclusive_scan(tiles * toks, tmp, &t2);
    block_exclusive_scan(toks, tmp, &t3);
    rowtok += t1;
    tiletok += t2;
    segtok += t3;
  }
  if (threadIdx.x == 0) {
    const long long work = (long long)tiletok * v.Hkv;              // tile-tokens over all heads
    const long long target_units = (long long)GB_SEG_UNITS_PCT * (v.num_sms > 0 ? v.num_sms : 1) / 100;
    int split = (int)(((work + target_units - 1) / target_units + 127) / 128 * 128);
    const int max_tokens = v.max_pages * v.P;
    const int min_split = ((max_tokens + (kMaxSegRecords - kMaxSegDepth) - 1) / (kMaxSegRecords - kMaxSegDepth) + 127) /
                          128 * 128;
    split = max(split, max(128, min_split));
    s_split = split;
    v.ctl[kCtlSegSplit] = split;
    v.ctl[kCtlSegRowTok] = rowtok;
    v.ctl[kCtlSegTileTok] = tiletok;
    v.ctl[kCtlSegTok] = segtok;
  }
  __syncthreads();
  const int split = s_split;
  // Entries sorted by length (tiles of 128 tokens), longest first, so that the grouped
  // kernel's snake assignment of units to CTAs balances the work: count entries per
  // length, lay the lengths out in descending order, then scatter.
  const int full_len = split / 128;
  for (int i = threadIdx.x; i < kSegLenBuckets; i += blockDim.x) hist[i] = 0;
  __syncthreads();
  for (int sidx = threadIdx.x; sidx < nseg; sidx += blockDim.x) {
    const int tiles = (v.seg_g[sidx] * v.G + rows_per_tile - 1) / rows_per_tile;
    const int toks = v.seg_len[sidx] * v.P;
    const int splits = (toks + split - 1) / split;
    v.seg_splits[sidx] = splits;
    const int last_len = min((toks - (splits - 1) * split + 127) / 128, kSegLenBuckets - 1);
    if (splits > 1) atomicAdd(&hist[min(full_len, kSegLenBuckets - 1)], tiles * (splits - 1));
    atomicAdd(&hist[last_len], tiles);
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    int acc = 0;
    for (int b = kSegLenBuckets - 1; b >= 0; --b) {  // longest first
      const int c = hist[b];
      hist[b] = acc;
      acc += c;
    }
    s_total = acc;
  }
  __syncthreads();
  const int carry = s_total;
  for (int sidx = threadIdx.x; sidx < nseg; sidx += blockDim.x) {
    const int tiles = (v.seg_g[sidx] * v.G + rows_per_tile - 1) / rows_per_tile;
    const int toks = v.seg_len[sidx] * v.P;
    const int splits = v.seg_splits[sidx];
    for (int sp = 0; sp < splits; ++sp) {
      const int len = min((min(toks - sp * split, split) + 127) / 128, kSegLenBuckets - 1);
      const int e0 = atomicAdd(&hist[len], tiles);
      for (int t = 0; t < tiles; ++t) {
        const int e = e0 + t;
        if (e < cap) {
          v.seg_tile_seg[e] = sidx;
          v.seg_tile_t[e] = t;
          v.seg_tile_split[e] = sp;
        }
      }
    }
  }
  __syncthreads();
  // The list holds at most 9 * max_beams + 2 * SMs entries (each beam sits in at most
  // kMaxSegDepth segments of >= 2 sharers) and a beam at most kMaxSegDepth + 32 records,
  // so neither limit is reached for pools of 8 beams or more.  Should the list still
  // overflow, the step is left entirely to the per-beam path.
  const bool overflow = carry > cap;
  for (int b = threadIdx.x; b < v.max_beams; b += blockDim.x) {
    int off = 0;
    for (int k = 0; k < v.seg_nseg[b]; ++k) {
      v.seg_rec_off[b * kMaxSegDepth + k] = off;
      off += v.seg_splits[v.seg_bid[b * kMaxSegDepth + k]];
    }
    if (overflow || off > kMaxSegRecords) {
      v.seg_cover[b] = 0;
      v.seg_nseg[b] = 0;
      off = 0;
    }
    v.seg_nrec[b] = off;
  }
  if (threadIdx.x == 0) v.ctl[kCtlSegTiles] = overflow ? 0 : carry;
}

cudaError_t rebuild_segments(gb_pool* pool, cudaStream_t s) {
  const PoolView& v = pool->view;
  if (!v.grouped) return cudaSuccess;
  const unsigned long long gen = ++pool->seg_gen;
  const int warps_per_block = 8;
  cudaError_t e = launch_pdl(k_seg_scan, (v.max_beams + warps_per_block - 1) / warps_per_block,
                             warps_per_block * 32, 0, s, v, gen);
  const int n = v.max_beams * kMaxSegDepth;
  if (e == cudaSuccess) e = launch_pdl(k_seg_lead, (n + 255) / 256, 256, 0, s, v, gen);
  if (e == cudaSuccess) e = launch_pdl(k_seg_members, (n + 255) / 256, 256, 0, s, v);
  if (e == cudaSuccess) e = launch_pdl(k_seg_tiles, 1, 1024, 0, s, v);
  pool->launches += 4;
  return e;
}

}  // namespace gb
