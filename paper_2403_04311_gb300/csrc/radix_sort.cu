// Stable LSD radix sort of (u32 key, u32 value) pairs, onesweep style
// (Adinets & Merrill, "Onesweep: A Faster Least Significant Digit Radix Sort
// for GPUs", 2022), written for this library:
//  * one upfront pass builds the digit histograms of every pass at once, with
//    warp-aggregated shared-memory counts (__match_any_sync picks one leader
//    per distinct digit in the warp);
//  * each pass is ONE kernel: a CTA ranks its 4096-key tile with match.any +
//    popc per warp, publishes per-digit tile counts, resolves its global
//    digit offsets by decoupled look-back over earlier tiles (bounded wait),
//    stages the tile in shared memory in digit order and writes it out in
//    runs of equal digits;
//  * tiles come from an atomic counter, so waits only target running CTAs.
// Key bits per pass: 8.  The element count is read on the device, so the
// sort can follow a device-computed size without a host round trip.
#include "common.cuh"
#include "kernels.h"
#include "scan.cuh"

namespace alto {

constexpr int kSortThreads = 256;
constexpr int kSortItems = 16;
constexpr int kSortTile = kSortThreads * kSortItems;  // 4096
constexpr int kRadix = 256;
constexpr u32 kSmallSort = 8192;  // at most this many pairs: the one-CTA sort

__global__ void __launch_bounds__(256) k_sort_hist(const u32* n_dev, u32 n_cap, const u32* keys,
                                                   int passes, u32* hist, Ctl* ctl) {
  pdl_enter();
  __shared__ u32 sh[4][kRadix];
  for (int i = threadIdx.x; i < 4 * kRadix; i += blockDim.x) (&sh[0][0])[i] = 0;
  __syncthreads();
  u32 n = halted(ctl) ? 0 : min(*n_dev, n_cap);
  const int lane = threadIdx.x & 31;
  const u32 stride = gridDim.x * blockDim.x;
  for (u32 wbase = (blockIdx.x * blockDim.x + (threadIdx.x & ~31u)); wbase < n; wbase += stride) {
    u32 i = wbase + lane;
    bool valid = i < n;
    u32 k = valid ? keys[i] : 0;
    for (int p = 0; p < passes; ++p) {
      u32 d = valid ? ((k >> (8 * p)) & 255u) : 256u;
      u32 peers = __match_any_sync(0xFFFFFFFFu, d);
      if (valid && lane == __ffs(peers) - 1) atomicAdd(&sh[p][d], (u32)__popc(peers));
    }
  }
  __syncthreads();
  for (int i = threadIdx.x; i < passes * kRadix; i += blockDim.x) {
    u32 c = (&sh[0][0])[i];
    if (c) atomicAdd(hist + i, c);
  }
}

// Exclusive scan of each pass's 256 digit counts; clears the histogram.
__global__ void __launch_bounds__(256) k_sort_binbase(u32* hist, u32* bin_base, int passes) {
  pdl_enter();
  __shared__ u32 s_w[kWarps];
  const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
  for (int p = 0; p < passes; ++p) {
    u32 c = hist[p * kRadix + t];
    u32 x = c;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      u32 y = __shfl_up_sync(0xFFFFFFFFu, x, o);
      if (lane >= o) x += y;
    }
    if (lane == 31) s_w[warp] = x;
    __syncthreads();
    u32 pre = 0;
    for (int w = 0; w < warp; ++w) pre += s_w[w];
    bin_base[p * kRadix + t] = pre + x - c;
    hist[p * kRadix + t] = 0;
    __syncthreads();
  }
}

__device__ __forceinline__ u32 block_excl_scan256(u32 v, u32* s_w) {
  const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
  u32 x = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    u32 y = __shfl_up_sync(0xFFFFFFFFu, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) s_w[warp] = x;
  __syncthreads();
  u32 pre = 0;
  for (int w = 0; w < warp; ++w) pre += s_w[w];
  __syncthreads();
  return pre + x - v;
}

__global__ void __launch_bounds__(kSortThreads) k_onesweep(const u32* n_dev, u32 n_cap, const u32* kin,
                                                           const u32* vin, u32* kout, u32* vout,
                                                           int shift, const u32* bin_base, u64* lb,
                                                           u64 lb_tiles, Ctl* ctl, int site,
                                                           u64 spin_limit) {
  pdl_enter();
  __shared__ u32 whist[kWarps][kRadix];
  __shared__ u32 s_k[kSortTile];
  __shared__ u32 s_v[kSortTile];
  __shared__ u32 s_toff[kRadix];
  __shared__ u32 s_gbase[kRadix];
  __shared__ u32 s_w[kWarps];
  __shared__ u32 s_tile;
  const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
  const u32 n = halted(ctl) ? 0 : min(*n_dev, n_cap);
  u32 ntiles = (n + kSortTile - 1) / kSortTile;
  if (ntiles > lb_tiles) ntiles = (u32)lb_tiles;
  const u32 es = epoch_site(ctl, site);
  for (;;) {
    if (t == 0) s_tile = take_tile(ctl, site);
    for (int i = t; i < kWarps * kRadix; i += kSortThreads) (&whist[0][0])[i] = 0;
    __syncthreads();
    const u32 tile = s_tile;
    if (tile >= ntiles) break;
    const u32 wbase = tile * kSortTile + warp * (kSortItems * 32);
    u32 keys[kSortItems];
    u32 rank[kSortItems];
    // issue every load of the tile before ranking
#pragma unroll
    for (int r = 0; r < kSortItems; ++r) {
      const u32 idx = wbase + r * 32 + lane;
      keys[r] = (idx < n) ? __ldcs(kin + idx) : 0u;
    }
#pragma unroll
    for (int r = 0; r < kSortItems; ++r) {
      u32 idx = wbase + r * 32 + lane;
      bool valid = idx < n;
      u32 k = keys[r];
      u32 d = valid ? ((k >> shift) & 255u) : 256u;
      u32 peers = __match_any_sync(0xFFFFFFFFu, d);
      int leader = __ffs(peers) - 1;
      u32 old = 0;
      if (valid && lane == leader) {
        old = whist[warp][d];
        whist[warp][d] = old + __popc(peers);
      }
      old = __shfl_sync(0xFFFFFFFFu, old, leader);
      rank[r] = old + __popc(peers & lanemask_lt());
      __syncwarp();
    }
    __syncthreads();
    // digit t: exclusive offsets across warps and the tile's count
    u32 cnt = 0;
#pragma unroll
    for (int w = 0; w < kWarps; ++w) {
      u32 c = whist[w][t];
      whist[w][t] = cnt;
      cnt += c;
    }
    // decoupled look-back for digit t
    u32 excl = 0;
    volatile u64* slot = lb + (u64)tile * kRadix + t;
    if (tile == 0) {
      *slot = ((u64)es << 34) | (2ull << 32) | cnt;
    } else {
      *slot = ((u64)es << 34) | (1ull << 32) | cnt;
      long long pred = (long long)tile - 1;
      u64 spins = 0;
      const bool stall = ctl->test_stall != 0;  // test hook: nothing is ever published
      while (pred >= 0) {
        volatile u64* ps = lb + (u64)pred * kRadix + t;
        u64 v = *ps;
        u32 kind = (u32)(v >> 32) & 3u;
        if ((u32)(v >> 34) != es || kind == 0 || stall) {
          if (++spins > spin_limit || *(volatile int*)&ctl->abort) {
            raise_timeout(ctl);
            break;
          }
          continue;
        }
        excl += (u32)v;
        if (kind == 2u) break;
        --pred;
      }
      *slot = ((u64)es << 34) | (2ull << 32) | (excl + cnt);
    }
    u32 toff = block_excl_scan256(cnt, s_w);
    s_toff[t] = toff;
    s_gbase[t] = bin_base[t] + excl - toff;
    __syncthreads();
#pragma unroll
    for (int r = 0; r < kSortItems; ++r) {
      u32 idx = wbase + r * 32 + lane;
      if (idx < n) {
        u32 d = (keys[r] >> shift) & 255u;
        u32 p = s_toff[d] + whist[warp][d] + rank[r];
        s_k[p] = keys[r];
        s_v[p] = vin ? __ldcs(vin + idx) : idx;
      }
    }
    __syncthreads();
    const u32 cnt_tile = min((u32)kSortTile, n - tile * kSortTile);
    for (u32 p = t; p < cnt_tile; p += kSortThreads) {
      u32 k = s_k[p];
      u32 g = s_gbase[(k >> shift) & 255u] + p;
      if (g < n) {
        kout[g] = k;
        vout[g] = s_v[p];
      }
    }
    __syncthreads();
  }
  if (t == 0) finish_ctas(ctl, site, &ctl->exit_ctr[site]);
}

// Up to kSmallSort pairs: the whole sort in one CTA, every pass in shared
// memory.  The 32 warps own contiguous runs of 256 elements in index order
// and rank a round of 32 with match.any + popc, as a tile of the onesweep
// does; the digit offsets come from the per-warp counts with no look-back.
// The result lands in the buffer the onesweep passes would have left it in.
constexpr int kSmallSortThreads = 1024;
constexpr u32 kSmallSortWarps = kSmallSortThreads / 32;
constexpr u32 kSmallSortItems = kSmallSort / kSmallSortThreads;  // 8 a thread
constexpr size_t kSmallSortSmem = (size_t)4 * kSmallSort * sizeof(u32) + (size_t)kSmallSortWarps * kRadix * sizeof(u32);

__global__ void __launch_bounds__(kSmallSortThreads) k_sort_small(const u32* n_dev, u32 n_cap, u32* k0, u32* v0,
                                                                  u32* kres, u32* vres, int passes,
                                                                  bool vals_identity, Ctl* ctl) {
  pdl_enter();
  extern __shared__ u32 smem[];
  u32* sk[2] = {smem, smem + kSmallSort};
  u32* sv[2] = {smem + 2 * kSmallSort, smem + 3 * kSmallSort};
  u32(*whist)[kRadix] = reinterpret_cast<u32(*)[kRadix]>(smem + 4 * kSmallSort);
  __shared__ u32 s_base[kRadix];
  __shared__ u32 s_w[8];
  const u32 n = halted(ctl) ? 0 : min(min(*n_dev, n_cap), kSmallSort);
  const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
  for (u32 i = t; i < n; i += kSmallSortThreads) {
    sk[0][i] = k0[i];
    sv[0][i] = vals_identity ? i : v0[i];
  }
  int cur = 0;
  for (int p = 0; p < passes; ++p) {
    const int shift = 8 * p;
    for (u32 i = t; i < kSmallSortWarps * kRadix; i += kSmallSortThreads) (&whist[0][0])[i] = 0;
    __syncthreads();
    u32 keys[kSmallSortItems], rank[kSmallSortItems];
    const u32 wbase = (u32)warp * (kSmallSortItems * 32);
#pragma unroll
    for (u32 r = 0; r < kSmallSortItems; ++r) {
      const u32 idx = wbase + r * 32 + lane;
      const bool valid = idx < n;
      const u32 k = valid ? sk[cur][idx] : 0u;
      keys[r] = k;
      const u32 d = valid ? ((k >> shift) & 255u) : 256u;
      const u32 peers = __match_any_sync(0xFFFFFFFFu, d);
      const int leader = __ffs(peers) - 1;
      u32 old = 0;
      if (valid && lane == leader) {
        old = whist[warp][d];
        whist[warp][d] = old + __popc(peers);
      }
      old = __shfl_sync(0xFFFFFFFFu, old, leader);
      rank[r] = old + __popc(peers & lanemask_lt());
      __syncwarp();
    }
    __syncthreads();
    // digit t (threads 0..255): exclusive offsets across warps, then across digits
    u32 cnt = 0;
    if (t < kRadix) {
      for (u32 w = 0; w < kSmallSortWarps; ++w) {
        const u32 c = whist[w][t];
        whist[w][t] = cnt;
        cnt += c;
      }
    }
    {
      u32 x = cnt;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const u32 y = __shfl_up_sync(0xFFFFFFFFu, x, o);
        if (lane >= o) x += y;
      }
      if (t < kRadix && lane == 31) s_w[warp] = x;
      __syncthreads();
      if (t < kRadix) {
        u32 pre = 0;
        for (int w = 0; w < warp; ++w) pre += s_w[w];
        s_base[t] = pre + x - cnt;
      }
    }
    __syncthreads();
#pragma unroll
    for (u32 r = 0; r < kSmallSortItems; ++r) {
      const u32 idx = wbase + r * 32 + lane;
      if (idx < n) {
        const u32 d = (keys[r] >> shift) & 255u;
        const u32 pos = s_base[d] + whist[warp][d] + rank[r];
        sk[cur ^ 1][pos] = keys[r];
        sv[cur ^ 1][pos] = sv[cur][idx];
      }
    }
    __syncthreads();
    cur ^= 1;
  }
  for (u32 i = t; i < n; i += kSmallSortThreads) {
    kres[i] = sk[cur][i];
    vres[i] = sv[cur][i];
  }
}

cudaError_t sort_prepare() {
  return cudaFuncSetAttribute(k_sort_small, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmallSortSmem);
}

int sort_pairs(const u32* n_dev, u32 n_cap, int bits, bool vals_identity, SortBuffers& b,
               Ctl* ctl, int site_base, u64 spin_limit, int num_sms, cudaStream_t s,
               int* launches) {
  int passes = (bits + 7) / 8;
  if (passes < 1) passes = 1;
  if (passes > 4) passes = 4;
  const int res = passes & 1;  // the buffers the passes leave the result in
  int nl = 0;
  if (n_cap <= kSmallSort) {
    // every count the capacity allows fits one CTA: one launch for the sort
    launch_pdl(k_sort_small, 1, kSmallSortThreads, kSmallSortSmem, s, n_dev, n_cap, b.keys[0], b.vals[0],
               b.keys[res], b.vals[res], passes, vals_identity, ctl);
    nl += 1;
  } else {
    u32 tiles_cap = (n_cap + kSortTile - 1) / kSortTile;
    if (tiles_cap == 0) tiles_cap = 1;
    int hist_grid = num_sms * 2;
    launch_pdl(k_sort_hist, hist_grid, 256, 0, s, n_dev, n_cap, b.keys[0], passes, b.hist, ctl);
    launch_pdl(k_sort_binbase, 1, 256, 0, s, b.hist, b.bin_base, passes);
    // four CTAs per SM (one per SM measured slower: each CTA then takes about
    // two tiles in turn, and a tile's look-back waits on the one before)
    u32 g4 = (u32)num_sms * 4u;
    int grid = (int)(tiles_cap < g4 ? tiles_cap : g4);
    int cur = 0;
    for (int p = 0; p < passes; ++p) {
      const u32* vin = (p == 0 && vals_identity) ? nullptr : b.vals[cur];
      launch_pdl(k_onesweep, grid, kSortThreads, 0, s, n_dev, n_cap, b.keys[cur], vin, b.keys[cur ^ 1],
                 b.vals[cur ^ 1], 8 * p, b.bin_base + p * kRadix, b.lookback, b.lb_tiles, ctl, site_base + p,
                 spin_limit);
      cur ^= 1;
    }
    nl += 2 + passes;
  }
  if (launches) *launches += nl;
  return res;
}

}  // namespace alto
