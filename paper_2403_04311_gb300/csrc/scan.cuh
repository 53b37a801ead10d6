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

constexpr int kScanThreads = 256;
constexpr int kScanItems = 8;
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

// Sum of everything before `tile`; serial walk by one thread.
__device__ __forceinline__ u64 lb_walk(LookbackState st, u32 tile, u32 es, Ctl* ctl, u64 spin_limit) {
  u64 excl = 0;
  long long pred = (long long)tile - 1;
  u64 spins = 0;
  while (pred >= 0) {
    volatile u32* fp = st.flag + pred;
    u32 f = *fp;
    if ((f >> 2) != es || (f & 3u) == 0) {
      if (++spins > spin_limit || *(volatile int*)&ctl->abort) {
        raise_timeout(ctl);
        break;
      }
      continue;
    }
    __threadfence();
    const bool inclusive = (f & 3u) == 2u;
    volatile u64* vp = (inclusive ? st.inc : st.agg) + pred;
    excl += *vp;
    if (inclusive) break;
    --pred;
  }
  return excl;
}

template <class F>
__global__ void __launch_bounds__(kScanThreads) k_scan(F f, LookbackState st, Ctl* ctl, int site,
                                                       u32* exit_ctr, u64 spin_limit) {
  __shared__ u32 s_tile;
  __shared__ u64 s_warp[kWarps];
  __shared__ u64 s_excl;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const u64 n = halted(ctl) ? 0 : f.size(ctl);
  u64 ntiles = (n + kScanTile - 1) / kScanTile;
  if (ntiles == 0) ntiles = 1;
  if (ntiles > st.tiles) {  // capacity guard; the size itself is checked by the producer
    ntiles = st.tiles;
  }
  const u32 es = epoch_site(ctl, site);
  for (;;) {
    if (threadIdx.x == 0) s_tile = take_tile(ctl, site);
    __syncthreads();
    const u32 tile = s_tile;
    __syncthreads();
    if (tile >= ntiles) break;
    const u64 base = (u64)tile * kScanTile + (u64)threadIdx.x * kScanItems;
    u64 v[kScanItems];
    u64 sum = 0;
#pragma unroll
    for (int k = 0; k < kScanItems; ++k) {
      u64 i = base + k;
      v[k] = (i < n) ? f.value(i) : 0;
      sum += v[k];
    }
    u64 x = sum;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      u64 y = __shfl_up_sync(0xFFFFFFFFu, x, o);
      if (lane >= o) x += y;
    }
    if (lane == 31) s_warp[warp] = x;
    __syncthreads();
    u64 wpre = 0, agg = 0;
#pragma unroll
    for (int w = 0; w < kWarps; ++w) {
      u64 t = s_warp[w];
      if (w < warp) wpre += t;
      agg += t;
    }
    if (threadIdx.x == 0) {
      u64 excl = 0;
      if (tile == 0) {
        lb_publish(st, tile, es, 2u, agg);
      } else {
        lb_publish(st, tile, es, 1u, agg);
        excl = lb_walk(st, tile, es, ctl, spin_limit);
        lb_publish(st, tile, es, 2u, excl + agg);
      }
      s_excl = excl;
      if (tile == ntiles - 1) f.total(ctl, excl + agg);
    }
    __syncthreads();
    u64 run = s_excl + wpre + (x - sum);
#pragma unroll
    for (int k = 0; k < kScanItems; ++k) {
      u64 i = base + k;
      if (i < n) f.out(i, run, v[k]);
      run += v[k];
    }
    __syncthreads();
  }
  if (threadIdx.x == 0) finish_ctas(ctl, site, exit_ctr);
}

}  // namespace alto
