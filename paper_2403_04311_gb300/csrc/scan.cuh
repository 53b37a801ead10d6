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
// Scans of at most this many tiles run in the launch's first CTA alone, tile
// after tile with a running carry: no look-back, no tile or exit counters
// (the other CTAs return at once).  Small batches' scans are a tile or two,
// and there the counters and descriptors of a look-back cost more than the
// scan itself.
constexpr u32 kScanSmallTiles = 2;

// One 16-byte descriptor per tile, {value, epoch_site << 2 | kind} with kind
// 1 = the tile's own sum, 2 = the sum of tiles 0..t.  It is written and read
// with single 16-byte vector accesses, so a reader sees the old or the new
// descriptor whole -- never a value with the other kind's flag -- and no
// fence is needed between value and flag.
struct LookbackState {
  ulonglong2* desc;  // [tiles]
  u64 tiles;         // capacity
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
  const u64 f = (u64)((es << 2) | kind);
  asm volatile("st.volatile.global.v2.u64 [%0], {%1, %2};" ::"l"(st.desc + tile), "l"(v), "l"(f)
               : "memory");
}

__device__ __forceinline__ ulonglong2 lb_read(LookbackState st, long long tile) {
  ulonglong2 r;
  asm volatile("ld.volatile.global.v2.u64 {%0, %1}, [%2];"
               : "=l"(r.x), "=l"(r.y)
               : "l"(st.desc + tile)
               : "memory");
  return r;
}

// Sum of everything before `tile`, found by warp 0: each lane reads four
// predecessors of a 128-tile window (lane l takes tiles top-l, top-l-32, ...).
// The nearest inclusive prefix ends the walk; only the tiles nearer than it
// must have published (their aggregates), so a slow tile further back does
// not hold this one up.
__device__ __forceinline__ u64 lb_walk_warp(LookbackState st, u32 tile, u32 es, Ctl* ctl,
                                            u64 spin_limit) {
  const int lane = threadIdx.x & 31;
  u64 excl = 0;
  long long top = (long long)tile - 1;
  u64 spins = 0;
  const bool stall = ctl->test_stall != 0;  // test hook: nothing is ever published
  while (top >= 0) {
    ulonglong2 dsc[4];
    int stop = 128, wait = 128;  // nearest inclusive, nearest unpublished
#pragma unroll
    for (int r = 0; r < 4; ++r) {
      const long long p = top - lane - 32 * r;
      dsc[r] = make_ulonglong2(0, 0);
      u32 kind = 2;  // before tile 0: an inclusive prefix of 0
      if (p >= 0) {
        dsc[r] = lb_read(st, p);
        const u32 f = (u32)dsc[r].y;
        kind = ((f >> 2) == es && !stall) ? (f & 3u) : 0u;
      }
      const u32 inc = __ballot_sync(0xFFFFFFFFu, kind == 2u);
      const u32 unp = __ballot_sync(0xFFFFFFFFu, kind == 0u);
      if (inc && stop == 128) stop = 32 * r + __ffs(inc) - 1;
      if (unp && wait == 128) wait = 32 * r + __ffs(unp) - 1;
    }
    if (wait < stop) {
      if (++spins > spin_limit || *(volatile int*)&ctl->abort) {
        if (lane == 0) raise_timeout(ctl);
        break;
      }
      // back off: every waiting warp polls the same few lines of descriptors
      __nanosleep(64);
      continue;
    }
    u64 v = 0;
#pragma unroll
    for (int r = 0; r < 4; ++r) {
      const int dist = lane + 32 * r;
      const long long p = top - dist;
      if (p >= 0 && dist <= stop) v += dsc[r].x;
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xFFFFFFFFu, v, o);
    excl += v;
    if (stop < 128) break;
    top -= 128;
  }
  return excl;
}

// A tile's values are read in striped order (coalesced) into shared memory;
// each thread then owns kScanItems consecutive elements: a serial sum, one
// warp scan of the thread sums, one pass over the warp sums.  The thread
// writes its elements' tile-local exclusive prefixes back into shared memory
// so that the out() calls run in striped order too (coalesced stores).
// Element values fit in 32 bits (counts, lengths, flags); prefixes are
// 64-bit, tile-local prefixes 32-bit (a tile whose sum does not fit takes the
// blocked order instead).  Shared memory is padded by one word per 32 so that
// both access orders are free of bank conflicts.
//
// The look-back is one warp's job; the CTA's other warps would wait for it at
// a barrier.  Instead, once the tile's aggregate is published, every thread
// loads the NEXT tile's values into registers, so that those loads are in
// flight while warp 0 walks back (value() only reads the scan's inputs).  The
// next tile's id is taken one tile ahead for the same reason.
__device__ __forceinline__ u32 scan_pad(u32 p) { return p + (p >> 5); }

template <class F>
__device__ __forceinline__ void scan_load(const F& f, u64 n, u32 tile, u32 ntiles, u32 (&r)[kScanItems]) {
  const int t = threadIdx.x;
  const u64 base = (u64)tile * kScanTile;
#pragma unroll
  for (int k = 0; k < kScanItems; ++k) {
    const u64 i = base + (u64)(k * kScanThreads + t);
    r[k] = (tile < ntiles && i < n) ? (u32)f.value(i) : 0u;
  }
}

template <class F>
__device__ __forceinline__ void scan_body(const F& f, LookbackState st, Ctl* ctl, int site,
                                          u32* exit_ctr, u64 spin_limit) {
  __shared__ u32 s_next;
  __shared__ u32 s_v[kScanTile + kScanTile / 32];
  __shared__ u64 s_w[kScanWarps];
  __shared__ u64 s_excl;
  const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
  const u64 n = halted(ctl) ? 0 : f.size(ctl);
  u64 ntiles64 = (n + kScanTile - 1) / kScanTile;
  if (ntiles64 == 0) ntiles64 = 1;
  if (ntiles64 > st.tiles) ntiles64 = st.tiles;
  const u32 ntiles = (u32)ntiles64;
  const u32 es = epoch_site(ctl, site);
  // every CTA reads the same n, so all take the same path
  const bool small = ntiles <= kScanSmallTiles;
  if (small && blockIdx.x != 0) return;
  __shared__ u64 s_carry;  // small path: sum of the tiles before this one
  if (t == 0) {
    s_next = small ? 0u : take_tile(ctl, site);
    s_carry = 0;
  }
  __syncthreads();
  u32 tile = s_next;
  __syncthreads();
  u32 r[kScanItems];
  scan_load(f, n, tile, ntiles, r);
  while (tile < ntiles) {
    if (t == 0) s_next = small ? tile + 1 : take_tile(ctl, site);  // read after the barriers below
#pragma unroll
    for (int k = 0; k < kScanItems; ++k) s_v[scan_pad((u32)(k * kScanThreads + t))] = r[k];
    __syncthreads();
    const u64 base = (u64)tile * kScanTile;
    u32 w[kScanItems];
    u64 sum = 0;
#pragma unroll
    for (int k = 0; k < kScanItems; ++k) {
      w[k] = s_v[scan_pad((u32)(t * kScanItems + k))];
      sum += w[k];
    }
    u64 x = sum;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const u64 y = __shfl_up_sync(0xFFFFFFFFu, x, o);
      if (lane >= o) x += y;
    }
    if (lane == 31) s_w[warp] = x;
    __syncthreads();
    const u32 next = s_next;
    u64 wpre = 0, agg = 0;
#pragma unroll
    for (int q = 0; q < kScanWarps; ++q) {
      const u64 c = s_w[q];
      if (q < warp) wpre += c;
      agg += c;
    }
    const bool narrow = agg < (1ull << 32);
    u64 rel = wpre + (x - sum);  // tile-local exclusive prefix of this thread's first element
    if (narrow) {
#pragma unroll
      for (int k = 0; k < kScanItems; ++k) {
        s_v[scan_pad((u32)(t * kScanItems + k))] = (u32)rel;
        rel += w[k];
      }
    }
    if (!small && warp == 0 && lane == 0) lb_publish(st, tile, es, tile == 0 ? 2u : 1u, agg);
    // the next tile's loads go out while warp 0 walks back
    scan_load(f, n, next, ntiles, r);
    if (warp == 0) {
      u64 excl = 0;
      if (small) {
        excl = s_carry;
      } else if (tile != 0) {
        excl = lb_walk_warp(st, tile, es, ctl, spin_limit);
        if (lane == 0) lb_publish(st, tile, es, 2u, excl + agg);
      }
      if (lane == 0) {
        s_excl = excl;
        if (small) s_carry = excl + agg;
        if (tile == ntiles - 1) f.total(ctl, excl + agg);
      }
    }
    __syncthreads();
    const u64 ex0 = s_excl;
    if (narrow) {
#pragma unroll
      for (int k = 0; k < kScanItems; ++k) {
        const u32 p = (u32)(k * kScanThreads + t);
        const u64 i = base + p;
        const u32 r0 = s_v[scan_pad(p)];
        const u32 r1 = (p + 1 < (u32)kScanTile) ? s_v[scan_pad(p + 1)] : (u32)agg;
        if (i < n) f.out(i, ex0 + r0, (u64)(r1 - r0));
      }
    } else {
      u64 run = ex0 + wpre + (x - sum);
      const u64 first = base + (u64)t * kScanItems;
#pragma unroll
      for (int k = 0; k < kScanItems; ++k) {
        if (first + k < n) f.out(first + k, run, w[k]);
        run += w[k];
      }
    }
    __syncthreads();
    tile = next;
  }
  if (!small && t == 0) finish_ctas(ctl, site, exit_ctr);
}

template <class F>
__global__ void __launch_bounds__(kScanThreads, 2) k_scan(F f, LookbackState st, Ctl* ctl, int site,
                                                       u32* exit_ctr, u64 spin_limit) {
  pdl_enter();
  scan_body(f, st, ctl, site, exit_ctr, spin_limit);
}

// No work after the last CTA of a multi-scan launch.
struct NoLast {
  static constexpr bool kActive = false;
  static constexpr bool kSide = false;
  __device__ void operator()(Ctl*) const {}
};

// Three independent scans in one launch: blockIdx.y selects the scan, each
// with its own launch site (tile and exit counters) and look-back arrays.
// When L is active, the launch's last CTA to finish runs `last` once every
// scan's total is written (so a check of the totals needs no launch of its
// own); it must read what other CTAs wrote with volatile loads.  L::kSide
// selects the CTA counter of a launch that may run beside another one.
template <class F, class L>
__global__ void __launch_bounds__(kScanThreads, 2) k_scan3(F f0, F f1, F f2, LookbackState st0,
                                                        LookbackState st1, LookbackState st2,
                                                        Ctl* ctl, int site, u64 spin_limit, L last) {
  pdl_enter();
  const int y = blockIdx.y;
  // one inlined body per scan: selecting a functor at run time would copy it
  // to local memory
  if (y == 0) scan_body(f0, st0, ctl, site, &ctl->exit_ctr[site], spin_limit);
  else if (y == 1) scan_body(f1, st1, ctl, site + 1, &ctl->exit_ctr[site + 1], spin_limit);
  else scan_body(f2, st2, ctl, site + 2, &ctl->exit_ctr[site + 2], spin_limit);
  if (L::kActive && threadIdx.x == 0) {
    __threadfence();
    u32* ctr = L::kSide ? &ctl->last_ctr2 : &ctl->last_ctr;
    const u32 k = atomicAdd(ctr, 1u);
    if (k == gridDim.x * gridDim.y - 1) {
      *ctr = 0;
      __threadfence();
      last(ctl);
    }
  }
}

}  // namespace alto
