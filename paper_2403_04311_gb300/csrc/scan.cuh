// Single-pass exclusive scan with decoupled look-back (Merrill & Garland,
// "Single-pass Parallel Prefix Scan with Decoupled Look-back", 2016),
// written for this library: persistent CTAs take tiles from a counter, so a
// tile only ever waits on tiles already owned by running CTAs; every wait is
// capped and reports ALTO_ETIMEOUT instead of hanging.
//
// The element values and the consumer of the prefixes are supplied by a
// functor, so compaction, offset assignment and segment discovery fuse into
// the scan:
//   u64  size(const Ctl*)          number of elements (read on the device)
//   u64  value(u64 i)              element i
//   void out(u64 i, u64 excl, u64 v)   exclusive prefix of element i
//   void total(Ctl*, u64 t)        grand total (called once, also for size 0)
#pragma once

#include "common.cuh"

namespace alto {

constexpr int kScanThreads = 512;
constexpr int kScanItems = 8;
constexpr int kScanWarps = kScanThreads / 32;
constexpr int kScanTile = kScanThreads * kScanItems;

// A tile's aggregate and its inclusive prefix live in separate arrays: a
// reader that saw the "aggregate" flag must never pick up the inclusive value
// written later into the same place.
struct LookbackState {
  u32* flag;  // [tiles] epoch_site << 2 | kind (1 aggregate, 2 inclusive)
  u64* agg;   // [tiles] the tile's own sum
  u64* inc;   // [tiles] sum of tiles 0..t
  u64 tiles;  // capacity
};

__device__ __forceinline__ u32 epoch_site(const Ctl* ctl, int site) {
  return (ctl->epoch * (u32)kSites + (u32)site) & 0x3FFFFFFFu;
}

// Take the next tile for this CTA; returns >= ntiles when done.  The last CTA
// to finish resets the counters for the next launch at the same site.
__device__ __forceinline__ u32 take_tile(Ctl* ctl, int site) {
  return atomicAdd(&ctl->tile_ctr[site], 1u);
}

__device__ __forceinline__ void finish_ctas(Ctl* ctl, int site, u32* exit_ctr) {
  __threadfence();
  u32 e = atomicAdd(exit_ctr, 1u);
  if (e == gridDim.x - 1) {
    ctl->tile_ctr[site] = 0;
    *exit_ctr = 0;
  }
}

__device__ __forceinline__ void lb_publish(LookbackState st, u32 tile, u32 es, u32 kind, u64 v) {
  volatile u64* vp = (kind == 2u ? st.inc : st.agg) + tile;
  volatile u32* fp = st.flag + tile;
  *vp = v;
  __threadfence();
  *fp = (es << 2) | kind;
}

// Sum of everything before `tile`, found by warp 0: each lane reads one
// predecessor of a 32-tile window; the nearest inclusive prefix ends the walk.
__device__ __forceinline__ u64 lb_walk_warp(LookbackState st, u32 tile, u32 es, Ctl* ctl,
                                            u64 spin_limit) {
  const int lane = threadIdx.x & 31;
  u64 excl = 0;
  long long top = (long long)tile - 1;
  u64 spins = 0;
  while (top >= 0) {
    const long long p = top - lane;
    u32 f = 0;
    bool ready = true;
    if (p >= 0) {
      f = *((volatile u32*)st.flag + p);
      ready = ((f >> 2) == es) && ((f & 3u) != 0);
    }
    if (!__all_sync(0xFFFFFFFFu, ready)) {
      if (++spins > spin_limit || *(volatile int*)&ctl->abort) {
        if (lane == 0) raise_timeout(ctl);
        break;
      }
      continue;
    }
    __threadfence();
    const bool inc = (p < 0) || ((f & 3u) == 2u);
    const u32 inc_mask = __ballot_sync(0xFFFFFFFFu, inc);
    const int stop = inc_mask ? __ffs(inc_mask) - 1 : 32;  // nearest inclusive predecessor
    u64 v = 0;
    if (p >= 0 && lane <= stop) v = *((volatile u64*)((lane == stop) ? st.inc : st.agg) + p);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xFFFFFFFFu, v, o);
    excl += v;
    if (inc_mask) break;
    top -= 32;
  }
  return excl;
}

// Tile = kScanItems rows of kScanThreads consecutive elements; thread t owns
// column t, so every value()/out() call is coalesced across the warp.
template <class F>
__global__ void __launch_bounds__(kScanThreads) k_scan(F f, LookbackState st, Ctl* ctl, int site,
                                                       u32* exit_ctr, u64 spin_limit) {
  __shared__ u32 s_tile;
  __shared__ u64 s_w[kScanItems][kScanWarps];
  __shared__ u64 s_excl;
  const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
  const u64 n = halted(ctl) ? 0 : f.size(ctl);
  u64 ntiles = (n + kScanTile - 1) / kScanTile;
  if (ntiles == 0) ntiles = 1;
  if (ntiles > st.tiles) ntiles = st.tiles;
  const u32 es = epoch_site(ctl, site);
  for (;;) {
    if (t == 0) s_tile = take_tile(ctl, site);
    __syncthreads();
    const u32 tile = s_tile;
    if (tile >= ntiles) break;
    const u64 base = (u64)tile * kScanTile;
    u64 v[kScanItems], x[kScanItems];
#pragma unroll
    for (int k = 0; k < kScanItems; ++k) {
      const u64 i = base + (u64)k * kScanThreads + t;
      v[k] = (i < n) ? f.value(i) : 0;
      x[k] = v[k];
    }
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
#pragma unroll
      for (int k = 0; k < kScanItems; ++k) {
        const u64 y = __shfl_up_sync(0xFFFFFFFFu, x[k], o);
        if (lane >= o) x[k] += y;
      }
    }
    if (lane == 31) {
#pragma unroll
      for (int k = 0; k < kScanItems; ++k) s_w[k][warp] = x[k];
    }
    __syncthreads();
    // row totals and this warp's offset inside each row
    u64 row_pre = 0, agg = 0;
    u64 off[kScanItems];
#pragma unroll
    for (int k = 0; k < kScanItems; ++k) {
      u64 rt = 0, wp = 0;
#pragma unroll
      for (int w = 0; w < kScanWarps; ++w) {
        const u64 c = s_w[k][w];
        if (w < warp) wp += c;
        rt += c;
      }
      off[k] = row_pre + wp;
      row_pre += rt;
    }
    agg = row_pre;
    if (warp == 0) {
      u64 excl = 0;
      if (tile == 0) {
        if (lane == 0) lb_publish(st, tile, es, 2u, agg);
      } else {
        if (lane == 0) lb_publish(st, tile, es, 1u, agg);
        excl = lb_walk_warp(st, tile, es, ctl, spin_limit);
        if (lane == 0) lb_publish(st, tile, es, 2u, excl + agg);
      }
      if (lane == 0) {
        s_excl = excl;
        if (tile == ntiles - 1) f.total(ctl, excl + agg);
      }
    }
    __syncthreads();
    const u64 ex0 = s_excl;
#pragma unroll
    for (int k = 0; k < kScanItems; ++k) {
      const u64 i = base + (u64)k * kScanThreads + t;
      if (i < n) f.out(i, ex0 + off[k] + x[k] - v[k], v[k]);
    }
    __syncthreads();
  }
  if (t == 0) finish_ctas(ctl, site, exit_ctr);
}

}  // namespace alto
