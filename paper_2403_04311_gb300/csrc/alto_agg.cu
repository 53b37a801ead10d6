// alto_agg: batched re-aggregation of streamed fragments by nested ancestry
// (Alto, arxiv 2403.04311, Sec. 3.1-4.3) on one GB300 GPU.
//
// One push runs this stream-ordered pipeline (no host synchronisation):
//   ingest      validate offsets/scores; find-or-insert each fragment's
//               leaf-parent group (level D-1) in the open-group hash table
//                                                                       [Sec. 4.2]
//   leaf level  count complete children, last-flag and child-index checks,
//               ancestry consistency, max score, top-k; merge with the table
//               entry and test completion                               [Sec. 3.1]
//               - without TOPK: every fragment, in arrival order, adds itself
//                 to its group's 64-byte table record (warp-aggregated
//                 atomics) and flags a repeated leaf slot; one pass over the
//                 touched groups then merges and tests them
//               - with TOPK (or streaming release): a stable onesweep radix
//                 sort by table slot, a look-back scan for each group's run,
//                 and a reduce by eight lanes, a warp or a block per run
//                 (segmented top-k)                                     [Sec. 4.3]
//   levels      the groups present at level l become the items of level l-1,
//               in the same two forms, up to level 0                    [Sec. 4.2]
//   emit order  completed groups ranked by (completion seq, deeper first)
//   CONCAT      open groups: append their leaves to per-group arena vectors;
//               completing groups: place every child span at slot
//               dense_base + child_index, scan the lengths, gather the spans
//               into the output payload ring                     [Sec. 3.2, 3.3]
//               With the CONCAT level M above the leaf parent, a group of a
//               level between completes into one span of its parent's vectors
//               (gathered level by level, bottom-up) before level M gathers.
//   records     one record per completed group, top-k pairs; free entries
//   streaming   (optional) an open leaf-parent CONCAT group whose first
//               unreleased child came in the batch releases its run of
//               present children as a partial record, placed and gathered
//               like a completion; its buffer then drops those children [Sec. 3.2]
#include <cuda_runtime.h>

#include <algorithm>
#include <cstdio>
#include <cstring>
#include <mutex>
#include <new>
#include <vector>

#include "alto_agg.h"
#include "common.cuh"
#include "kernels.h"

#include "scan.cuh"

namespace alto {

constexpr int kThreads = 256;

struct Batch {
  const u64* tags;
  const u32* off;
  const int32_t* pay;
  const float* score;
  u32 n;
  u64 n_payload;
};

struct Scratch {
  u32* leaf_sort_keys0;  // ingest writes the table slot of each fragment here
  u32* up_sort_keys0;    // item lookups write here
  u32* leaf_keys;        // sorted leaf keys (set by the host after the sort)
  u32* leaf_perm;
  u32* leaf_seg_start;   // [n_max + 1]
  u32* leaf_seg_of;      // [n_max]
  u32* up_keys;
  u32* up_perm;
  u32* up_seg_start;     // [n_max + 1] sorted levels: segment starts; atomic levels: touched entries
  u32* up_list2;         // [n_max] atomic levels: touched entries (alternating with up_seg_start)
  u32* it_rep[2];        // items: representative fragment
  u32* it_cseq[2];       // items: done << 31 | completion seq (batch-local)
  u32* it_skey[2];       // items: largest score key of the child
  u32* seg_vb0;          // leaf segments: meta vector base (leaves)
  u32* seg_vb1;          // leaf segments: payload vector base (elements)
  u32* seg_carry;        // leaf segments: 1 to the arena, 2 placed densely, 3 both (a partial release)
  u32* leaf_pos;         // [n_max] sorted leaf j: payload offset inside its segment's buffered data
  u32* leaf_mrank;       // [n_max] streaming, segments 3: meta index among the buffered leaves, kNone if placed
  u32* mask;             // [n_max] bit (D-1-l): a level-l group completes at this seq
  u32* mblk;             // [n_max/32 + 1] completions at the seqs of each run of 32
  u32* prefix;           // [n_max/32 + 1] completions before each run of 32 seqs
  u32* done_e;           // [done_cap]
  u32* done_lvl;
  u32* done_cseq;
  u32* done_rank;
  u32* r_done;           // by rank
  u32* r_dense_n;
  u32* r_topk_n;
  u32* r_meta_n;
  u64* r_dense_base;
  u64* r_topk_off;
  u64* r_arena_base;
  u64* c_dense_base;     // [done_cap + 1] by done index: dense slots of levels M < l
  u64* c_arena_base;     // [done_cap + 1] by done index: their buffered spans
  uint4* dense;          // [dense_cap] {stamp, len, owner entry or kNone, position}
  u64* dst;              // [dense_cap + 1]
  u64* pairset;          // [ps_mask + 1]
  u64 ps_mask;
  u32 done_cap;
  // streaming release
  u32* done_part;        // [done_cap] a partial release (cleared by the records): 1, or 2 when
                         // children buffered by earlier batches were released (the buffer is compacted)
  u32* bm;               // [bm_cap] per-batch presence bitmaps of the groups that release
  u64 bm_cap;
  u32* big_seg;          // [depth][big_cap] segments longer than kBigSeg, per level
  u32 big_cap;
  u32* rel_seg;          // [n_max] streaming: small leaf segments whose groups release a run
  Batch* batch;          // [1] the push's batch, stored by k_begin (read by graph replays)
  // split placement (CONCAT at the leaf parent): the leaf parents ranked
  // among themselves
  u32* lblk;             // [n_max/32 + 1] leaf parents completing at the seqs of each run of 32
  u32* lprefix;          // [n_max/32 + 1] leaf parents completing before each run
  u32* l_done;           // [done_cap] by leaf rank: done index
  u32* l_dense_n;        // [done_cap] by leaf rank: children
  u32* l_meta_n;         // [done_cap] by leaf rank: buffered spans
  u64* l_dense_base;     // [done_cap + 1] by leaf rank: first dense slot
  u64* l_arena_base;     // [done_cap + 1] by leaf rank: first buffered span
};

struct Dev {
  Ctl* ctl;
  Table tab;
  Arena ar;
  Cfg cfg;
  Scratch sc;
  alto_record* out_rec;
  int32_t* out_pay;
  alto_topk_pair* out_topk;
  // Split placement (set per batch by the host): with CONCAT at the leaf
  // parent, the payload path of the leaf parents that complete (their ranks
  // among themselves, dense slots, placement, length scan, gather) runs on a
  // second stream beside the upper levels and the record scans.  Only leaf
  // parents carry payload, and their order among themselves is their
  // completion order, so the payload offsets need nothing from the levels
  // above.
  int split;
};

// The batch of the push.  Kernels launched one by one get it by value; in a
// replay of a push's captured CUDA graph (G) their parameters are those of
// the capture, and the batch is the copy the graph's first kernel stored.
template <bool G>
__device__ __forceinline__ Batch batch_of(const Batch& bv, const Dev& d) {
  if constexpr (G) {
    return *d.sc.batch;
  } else {
    return bv;
  }
}

__device__ __forceinline__ bool poisoned(const Ctl* c) { return halted(c); }
// Payload-moving kernels also stand down once the batch has any error: its
// outputs are undefined and its offsets may not be trustworthy.
__device__ __forceinline__ bool no_copy(const Ctl* c) {
  return halted(c) || *(const volatile int*)&c->batch_err != 0;
}
// A split placement's kernels stand down on the errors raised before the
// fork (the leaf finalize's snapshot), not on those the upper levels raise
// beside them: what they find then does not depend on timing.
__device__ __forceinline__ bool stand_down(const Dev& d, const Ctl* c) {
  return d.split ? (halted(c) || *(const volatile int*)&c->pre_err != 0) : no_copy(c);
}

__device__ __forceinline__ u32 gtid() { return blockIdx.x * blockDim.x + threadIdx.x; }
__device__ __forceinline__ u32 gstride() { return gridDim.x * blockDim.x; }

// A place in a list whose length is the global `counter`, for every lane with
// `want` (kNone for the others), with one atomic per warp: tens of thousands
// of single appends to one address a batch serialise in one L2 slice.  All 32
// lanes of the warp call it together.
__device__ __forceinline__ u32 warp_take(bool want, u32* counter) {
  const u32 m = __ballot_sync(0xFFFFFFFFu, want);
  if (m == 0) return kNone;
  const int leader = __ffs(m) - 1;
  u32 base = 0;
  if ((int)(threadIdx.x & 31) == leader) base = atomicAdd(counter, (u32)__popc(m));
  base = __shfl_sync(0xFFFFFFFFu, base, leader);
  return want ? base + __popc(m & lanemask_lt()) : kNone;
}

// The same with one atomic on `counter` per block (a few thousand warps each
// appending to one address serialise on it: about 0.65 ns an atomic on the
// GB300).  All threads of the block call it together; sh.cnt is zero on entry
// and on return.
struct BlockTake {
  u32 cnt;
  u32 base;
};
__device__ __forceinline__ u32 block_take(bool want, u32* counter, BlockTake& sh) {
  const int lane = threadIdx.x & 31;
  const u32 m = __ballot_sync(0xFFFFFFFFu, want);
  const int wl = __ffs(m) - 1;
  u32 wbase = 0;
  if (m != 0 && lane == wl) wbase = atomicAdd(&sh.cnt, (u32)__popc(m));
  __syncthreads();
  if (threadIdx.x == 0) {
    sh.base = sh.cnt ? atomicAdd(counter, sh.cnt) : 0u;
    sh.cnt = 0;
  }
  __syncthreads();
  if (m != 0) wbase = __shfl_sync(0xFFFFFFFFu, wbase, wl);
  return want ? sh.base + wbase + __popc(m & lanemask_lt()) : kNone;
}

// ---------------------------------------------------------------------------
// open-group hash table (linear probing; a slot index is the entry id)
// ---------------------------------------------------------------------------
// Find the entry of `key`, or insert it.  A slot is empty, deleted (a
// tombstone: its group was emitted) or holds a key.  The walk from the home
// slot ends at the key or at the first empty slot; a key is new when it has
// not been met by then, and it takes the first deleted slot of the walk if
// there was one, else that empty slot.  Taking deleted slots keeps a table
// sized near the groups open at once from filling with tombstones.
//
// Within one launch slots only go from empty or deleted to a key, so every
// thread inserting the same key aims at the same first free slot unless that
// slot was taken meanwhile, and then its compare-and-swap fails: the thread
// walks again from that slot (the slots before it hold other keys for good).
// No key is ever placed twice, and a walk only grows while other threads take
// free slots, so it ends.  A key lies within max_probe slots of home; a walk
// that reaches that distance with no free slot met finds the table full.
//
// `publish`: other threads of this launch may add to the new entry's batch
// accumulators and compare with its chain row as soon as the key is in
// place (the level kernels that add their items to the parent level).  The
// insert then leaves the accumulators and `touch` alone (they are clear in a
// free slot) and, once the chain row is written, sets the entry's ready flag
// with release order.  Without it (no adder in the launch) the whole record
// is written, which also brings its line into L2 for the next kernel.
__device__ u32 ht_find_or_insert(const Table& tab, u64 key, u64 up, Ctl* ctl, int* inserted,
                                  const u64* tags = nullptr, u64 n = 0, u32 rep = 0, int l = 0,
                                  bool publish = false) {
  const u32 home = (u32)mix64(key) & tab.mask;
  const u32 reach = (u32)tab.max_probe;  // at most the table size
  u32 h = home, dist = 0;
  u32 free_at = kNone;  // first deleted slot of the walk
  for (;;) {
    if (dist < reach) {
      const u64 cur = ((volatile u64*)tab.key)[h];
      if (cur == key) return h;
      if (cur == kTomb && free_at == kNone) free_at = h;
      if (cur != kEmpty) {
        h = (h + 1) & tab.mask;
        ++dist;
        continue;
      }
    } else if (free_at == kNone) {
      break;
    }
    // the key is not in the table: take the first free slot of the walk
    const u32 t = (free_at != kNone) ? free_at : h;
    const u64 want = (free_at != kNone) ? kTomb : kEmpty;
    const u64 prev = atomicCAS((unsigned long long*)&tab.key[t], (unsigned long long)want,
                               (unsigned long long)key);
    if (prev == want) {
      // up, last = none, nothing completed, accumulators clear
      uint4* hw = reinterpret_cast<uint4*>(tab.hot + t);
      hw[0] = make_uint4((u32)up, (u32)(up >> 32), kNone, 0);
      if (publish) {
        tab.hot[t].maxc1 = 0;
        tab.hot[t].smax = 0;
        tab.hot[t].done_epoch = 0;
      } else {
        hw[1] = make_uint4(0, 0, 0, 0);
        hw[2] = make_uint4(kNone, 0, 0, 0);
        hw[3] = make_uint4(0, 0, 0, 0);
      }
      if (tab.rel) tab.rel[t] = 0;
      if (tab.vec_n) {
        tab.vec_n[2 * (u64)t] = 0;
        tab.vec_n[2 * (u64)t + 1] = 0;
      }
      if (tags) {
        for (int q = 0; q < l; ++q) tab.chain[(u64)t * tab.chain_len + q] = tags[(u64)q * n + rep];
      }
      if (tags && l == tab.leaf_level) {
        ulonglong2* cb = reinterpret_cast<ulonglong2*>(tab.cbits + 4 * (u64)t);
        cb[0] = make_ulonglong2(0, 0);
        cb[1] = make_ulonglong2(0, 0);
      }
      // the chain row is written: finders of this launch may compare with it
      if (publish) asm volatile("st.release.gpu.global.u32 [%0], %1;" ::"l"(tab.ready + t), "r"(1u) : "memory");
      *inserted = 1;
      return t;
    }
    if (prev == key) return t;
    // another key took the slot: walk again from it (its distance from home
    // is below reach, so the subtraction does not wrap)
    h = t;
    dist = (t - home) & tab.mask;
    free_at = kNone;
  }
  // The table is full: the batch stops here.  The caller gets kNone and
  // stores entry 0 where an index is needed, so that nothing indexes out of
  // bounds; the abort keeps every later kernel of the batch from treating
  // entry 0 as this group (which would report false duplicates).
  raise_err(ctl, ALTO_ENOSPC);
  *(volatile int*)&ctl->abort = 1;
  return kNone;
}

// Batch-local set of (entry, child) slots; returns true if already present.
// Keys carry a 7-bit batch epoch so that old batches' keys read as free.
// (Placing a group's children in neighbouring slots was tried: the runs it
// builds lengthen every other probe, and the batch got 4x slower.)
__device__ bool ps_insert(const Scratch& sc, u32 e, u32 c, u32 ep7, Ctl* ctl) {
  const u64 k57 = ((u64)e << 31) | c;
  const u64 full = ((u64)ep7 << 57) | k57;
  u64 h = mix64(k57) & sc.ps_mask;
  for (int p = 0; p < 8192; ++p) {
    u64 cur = ((volatile u64*)sc.pairset)[h];
    if (cur == full) return true;
    if ((u32)(cur >> 57) != ep7) {
      u64 prev = atomicCAS((unsigned long long*)&sc.pairset[h], (unsigned long long)cur,
                           (unsigned long long)full);
      if (prev == cur) return false;
      if (prev == full) return true;
      continue;
    }
    h = (h + 1) & sc.ps_mask;
  }
  raise_err(ctl, ALTO_ENOSPC);
  return false;
}

// A leaf slot given twice.  Slots below 256 go through the leaf parent's
// bitmap, which lives as long as the open group (so a slot repeated in a later
// batch is caught too) and sits next to the group's other state in L2; the
// others through the batch-local pair set.  Only for launches after the one
// that inserted the entry (the insert clears the bitmap).
__device__ __forceinline__ bool leaf_dup(const Table& tab, const Scratch& sc, u32 e, u32 c, u32 ep7,
                                         Ctl* ctl) {
  if (c < 256) {
    const u64 bit = 1ull << (c & 63);
    const u64 old = atomicOr((unsigned long long*)&tab.cbits[4 * (u64)e + (c >> 6)], (unsigned long long)bit);
    return (old & bit) != 0;
  }
  return ps_insert(sc, e, c, ep7, ctl);
}

__device__ __forceinline__ bool chain_differs(const Table& tab, u32 e, const u64* tags, u64 n, u32 rep,
                                              int l) {
  // the chain row is padded to an even length: read it two tags at a time
  const ulonglong2* row = reinterpret_cast<const ulonglong2*>(tab.chain + (u64)e * tab.chain_len);
  bool bad = false;
  for (int q = 0; q < l; q += 2) {
    const ulonglong2 v = row[q >> 1];
    if (tags[(u64)q * n + rep] != v.x) bad = true;
    if (q + 1 < l && tags[(u64)(q + 1) * n + rep] != v.y) bad = true;
  }
  return bad;
}

__device__ __forceinline__ u32 epoch7(const Ctl* ctl) { return ((ctl->epoch - 1) % 127u) + 1u; }

// ---------------------------------------------------------------------------
// arena: per-group vectors made of geometrically growing chunks
// ---------------------------------------------------------------------------
__device__ __forceinline__ u64 vec_addr(const Table& tab, u32 e, int vec, u64 x, bool* ok) {
  int j = chunk_of(x);
  if (j >= kNumChunks) {
    *ok = false;
    return 0;
  }
  u32 base = tab.dir[((u64)e * kVecs + vec) * kNumChunks + j];
  *ok = base != kNone;
  return (u64)base + (x - chunk_start(j));
}

__device__ u32 alloc_chunk(const Arena& ar, Ctl* ctl, int j) {
  int old = atomicSub(&ctl->top[j], 1);
  if (old > 0) return ar.stack[ar.stack_off[j] + (u64)(old - 1)];
  u64 sz = chunk_size(j);
  u64 off = atomicAdd((unsigned long long*)&ctl->bump, (unsigned long long)sz);
  if (off + sz > ar.elems) {
    raise_err(ctl, ALTO_ENOSPC);
    return kNone;
  }
  return (u32)off;
}

__device__ void free_chunk(const Arena& ar, Ctl* ctl, int j, u32 chunk) {
  if (chunk == kNone) return;
  int pos = atomicAdd(&ctl->top[j], 1);
  if ((u64)pos < ar.stack_cap[j]) ar.stack[ar.stack_off[j] + (u64)pos] = chunk;
}

// Chunks for the growth of each requesting thread's two vectors of entry e:
// every class that starts in [old, new) of a vector (vector 0 holds two int32
// per leaf), with one free-stack atomic (and at most one bump atomic) per
// chunk class and block.  A stack may go negative; the record scans' last
// CTA (CapCheck) clears that before anything is freed.  All threads of the
// block call it together; the counters in `sh` are zero on entry and on
// return.
struct GrowShared {
  u32 cnt[kNumChunks];
  u32 rank[kNumChunks];
  int old[kNumChunks];
  u32 avail[kNumChunks];
  unsigned long long bump[kNumChunks];
  unsigned long long got;
};
__device__ void block_grow(const Table& tab, const Arena& ar, Ctl* ctl, bool want, u32 e, u64 old0,
                           u64 new0, u64 old1, u64 new1, GrowShared& sh) {
  int jf[kVecs], jl[kVecs];
  const u64 olds[kVecs] = {old0, old1}, news[kVecs] = {new0, new1};
#pragma unroll
  for (int v = 0; v < kVecs; ++v) {
    jf[v] = kNumChunks;
    jl[v] = -1;
    if (want && news[v] > olds[v]) {
      jf[v] = (olds[v] == 0) ? 0 : chunk_of(olds[v] - 1) + 1;
      jl[v] = chunk_of(news[v] - 1);
      if (jl[v] >= kNumChunks) {
        raise_err(ctl, ALTO_ENOSPC);
        jl[v] = kNumChunks - 1;
      }
    }
  }
#pragma unroll
  for (int v = 0; v < kVecs; ++v)
    for (int j = jf[v]; j <= jl[v]; ++j) atomicAdd(&sh.cnt[j], 1u);
  __syncthreads();
  if (threadIdx.x < kNumChunks) {
    const int j = threadIdx.x;
    const u32 cnt = sh.cnt[j];
    int old = 0;
    u32 avail = 0;
    unsigned long long bump = 0;
    if (cnt) {
      old = atomicSub(&ctl->top[j], (int)cnt);
      avail = (old <= 0) ? 0u : min((u32)old, cnt);
      if (cnt > avail)
        bump = atomicAdd((unsigned long long*)&ctl->bump, (unsigned long long)(cnt - avail) * chunk_size(j));
    }
    sh.old[j] = old;
    sh.avail[j] = avail;
    sh.bump[j] = bump;
  }
  __syncthreads();
  u64 got = 0;
#pragma unroll
  for (int v = 0; v < kVecs; ++v) {
    for (int j = jf[v]; j <= jl[v]; ++j) {
      const u32 r = atomicAdd(&sh.rank[j], 1u);
      u32 c;
      if (r < sh.avail[j]) {
        c = ar.stack[ar.stack_off[j] + (u64)(sh.old[j] - 1 - (int)r)];
      } else {
        const u64 o = sh.bump[j] + (u64)(r - sh.avail[j]) * chunk_size(j);
        if (o + chunk_size(j) > ar.elems) {
          raise_err(ctl, ALTO_ENOSPC);
          c = kNone;
        } else {
          c = (u32)o;
        }
      }
      tab.dir[((u64)e * kVecs + v) * kNumChunks + j] = c;
      if (c != kNone) got += chunk_size(j);
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) got += __shfl_xor_sync(0xFFFFFFFFu, got, o);
  if ((threadIdx.x & 31) == 0 && got) atomicAdd(&sh.got, (unsigned long long)got);
  __syncthreads();
  if (threadIdx.x < kNumChunks) {
    sh.cnt[threadIdx.x] = 0;
    sh.rank[threadIdx.x] = 0;
  }
  if (threadIdx.x == 0 && sh.got) {
    atomicAdd((unsigned long long*)&ctl->arena_used, sh.got);
    sh.got = 0;
  }
  __syncthreads();
}

// ---------------------------------------------------------------------------
// CONCAT at a level M above the leaf parent.  A group of a level l with
// M < l <= D-1 that completes becomes one child span of its parent: its
// concatenation is reserved at the end of the parent's vectors (one 64-bit
// atomic on the parent's cursor: span index and payload position together)
// and copied there later in the batch, so that a group of level M finds all
// its children's concatenations, in any order, in its own vectors.
// ---------------------------------------------------------------------------
constexpr u64 kPos40 = (1ull << 40) - 1;

// levels whose completed groups hand a span to their parent
__device__ __forceinline__ bool chain_level(const Cfg& c, int l) {
  return c.concat_level >= 0 && l > c.concat_level;
}
// levels whose groups receive their children's spans (the leaf parent buffers leaves instead)
__device__ __forceinline__ bool chain_parent(const Cfg& c, int l) {
  return c.concat_level >= 0 && l >= c.concat_level && l < c.depth - 1;
}

// Chunks of every class that starts in [old_el, new_el) of entry e's vector vec.
__device__ void grow_vec(const Table& tab, const Arena& ar, Ctl* ctl, u32 e, int vec, u64 old_el,
                         u64 new_el) {
  if (new_el <= old_el) return;
  const int jf = (old_el == 0) ? 0 : chunk_of(old_el - 1) + 1;
  const int jl = chunk_of(new_el - 1);
  if (jl >= kNumChunks) raise_err(ctl, ALTO_ENOSPC);
  u64 got = 0;
  for (int j = jf; j <= jl && j < kNumChunks; ++j) {
    const u32 c = alloc_chunk(ar, ctl, j);
    tab.dir[((u64)e * kVecs + vec) * kNumChunks + j] = c;
    if (c != kNone) got += chunk_size(j);
  }
  if (got) atomicAdd((unsigned long long*)&ctl->arena_used, (unsigned long long)got);
}

// A receiving group takes the spans its children reserved in earlier launches
// of this batch: chunks for the growth, then the new sizes.
__device__ void chain_sync(const Table& tab, const Arena& ar, Ctl* ctl, u32 e) {
  const u64 cu = tab.cur[e];
  const u64 n0 = cu >> 40, n1 = cu & kPos40;
  const u32 o0 = tab.vec_n[2 * (u64)e], o1 = tab.vec_n[2 * (u64)e + 1];
  if (n0 == o0 && n1 == o1) return;
  // the 24-bit span count and the 32-bit sizes must not wrap
  if (n0 >= (1ull << 23) || n1 >= (1ull << 32)) {
    raise_err(ctl, ALTO_ENOSPC);
    return;
  }
  grow_vec(tab, ar, ctl, e, 0, 2 * (u64)o0, 2 * n0);
  grow_vec(tab, ar, ctl, e, 1, o1, n1);
  tab.vec_n[2 * (u64)e] = (u32)n0;
  tab.vec_n[2 * (u64)e + 1] = (u32)n1;
}

// Completed group e (child c of parent entry P) reserves its `total` elements.
// A cursor is zeroed when its entry is freed, so a parent inserted in the same
// launch can take reservations at once.
__device__ __forceinline__ void chain_reserve(const Table& tab, u32 e, u32 P, u32 c, u64 total) {
  const u64 old = atomicAdd((unsigned long long*)&tab.cur[P], (unsigned long long)((1ull << 40) | total));
  tab.par[e] = P;
  tab.cidx[e] = c;
  tab.app[e] = old;
}

// ---------------------------------------------------------------------------
// kernels
// ---------------------------------------------------------------------------
// Every table record as a free slot has it: no last child, nothing
// completed, accumulators clear (acc_fmin = none).
__global__ void k_init_hot(Hot* hot, u64 T) {
  pdl_enter();
  for (u64 i = (u64)blockIdx.x * blockDim.x + threadIdx.x; i < T; i += (u64)gridDim.x * blockDim.x) {
    uint4* hw = reinterpret_cast<uint4*>(hot + i);
    hw[0] = make_uint4(0, 0, kNone, 0);
    hw[1] = make_uint4(0, 0, 0, 0);
    hw[2] = make_uint4(kNone, 0, 0, 0);
    hw[3] = make_uint4(0, 0, 0, 0);
  }
}

// Start of a push: store the batch for kernels that read it from device
// memory (graph replays), reset the output counters a drain handed out
// (`reset`), and clear the per-batch fields.
__global__ void k_begin(Ctl* ctl, Batch b, Batch* store, int reset) {
  pdl_enter();
  if (store) *store = b;
  if (reset) {
    ctl->rec_count = 0;
    ctl->pay_count = 0;
    ctl->topk_count = 0;
  }
  ctl->pay_base = ctl->pay_count;
  ctl->epoch += 1;
  ctl->batch_err = 0;
  ctl->n_done = 0;
  ctl->skip_dense = 0;
  ctl->skip_rec = 0;
  ctl->pre_err = 0;
  ctl->dense_total = ctl->arena_total = ctl->pay_total = ctl->topk_total = ctl->n_emit = 0;
  ctl->leaf_dense_total = ctl->leaf_arena_total = 0;
  ctl->bm_used = 0;
  ctl->n_rel = 0;
  for (int l = 0; l < kMaxDepth; ++l) ctl->n_big[l] = 0;
  for (int l = 0; l < kMaxDepth; ++l) ctl->n_segs[l] = 0;
  ctl->n = (ctl->status == ALTO_OK) ? b.n : 0u;
}

template <bool G>
__global__ void __launch_bounds__(kThreads) k_ingest(Dev d, Batch bv) {
  pdl_enter();
  const Batch b = batch_of<G>(bv, d);
  Ctl* ctl = d.ctl;
  if (poisoned(ctl)) return;
  __shared__ u32 s_ins;
  if (threadIdx.x == 0) s_ins = 0;
  __syncthreads();
  const int D = d.cfg.depth;
  const u32 ep7 = epoch7(ctl);
  const bool sorted_leaf = d.cfg.score_op[D - 1] == ALTO_SCORE_TOPK || d.cfg.stream_leaf;
  for (u32 i = gtid(); i < b.n; i += gstride()) {
    u32 o0 = b.off[i], o1 = b.off[i + 1];
    if (o1 < o0 || (u64)o1 > b.n_payload) raise_err(ctl, ALTO_EINVAL);
    if (d.cfg.has_score && is_nan_bits(__float_as_uint(b.score[i]))) raise_err(ctl, ALTO_EINVAL);
    u64 t = b.tags[(u64)(D - 1) * b.n + i];
    u64 up = (D > 1) ? b.tags[(u64)(D - 2) * b.n + i] : 0ull;
    int ins = 0;
    u32 e = ht_find_or_insert(d.tab, ((u64)(D - 1) << 32) | tag_pid(t), up, ctl, &ins, b.tags,
                              b.n, i, D - 1);
    if (ins) atomicAdd(&s_ins, 1u);
    d.sc.leaf_sort_keys0[i] = (e == kNone) ? 0u : e;
    if (e == kNone) continue;
    // the sorted (TOPK) leaf path checks leaf slots here, spread over the
    // whole grid (in the reduce, a hot group's checks would all fall to the
    // block that reduces its segment); the accumulate does otherwise
    if (sorted_leaf && ps_insert(d.sc, e, tag_child(t), ep7, ctl)) raise_err(ctl, ALTO_EDUP);
  }
  __syncthreads();
  if (threadIdx.x == 0 && s_ins) atomicAdd((unsigned long long*)&ctl->live_groups, (u64)s_ins);
}

// Items of level l are the level-(l+1) groups present in the batch.
template <bool G>
__global__ void __launch_bounds__(kThreads) k_items_lookup(Dev d, Batch bv, int l, int in_set) {
  pdl_enter();
  const Batch b = batch_of<G>(bv, d);
  Ctl* ctl = d.ctl;
  if (poisoned(ctl)) return;
  __shared__ u32 s_ins;
  if (threadIdx.x == 0) s_ins = 0;
  __syncthreads();
  const u32 ni = min(ctl->n_segs[l + 1], d.cfg.n_max);
  const u32 ep7 = epoch7(ctl);
  const u32* it_rep = d.sc.it_rep[in_set];
  for (u32 x = gtid(); x < ni; x += gstride()) {
    u32 rep = it_rep[x];
    u64 t = b.tags[(u64)l * b.n + rep];
    u64 up = (l > 0) ? b.tags[(u64)(l - 1) * b.n + rep] : 0ull;
    int ins = 0;
    u32 e = ht_find_or_insert(d.tab, ((u64)l << 32) | tag_pid(t), up, ctl, &ins, b.tags, b.n, rep, l);
    if (ins) atomicAdd(&s_ins, 1u);
    d.sc.up_sort_keys0[x] = (e == kNone) ? 0u : e;
    if (e == kNone) continue;
    if (ps_insert(d.sc, e, tag_child(t), ep7, ctl)) raise_err(ctl, ALTO_EINCONSIST);
  }
  __syncthreads();
  if (threadIdx.x == 0 && s_ins) atomicAdd((unsigned long long*)&ctl->live_groups, (u64)s_ins);
}

// Segment discovery over sorted keys: seg_start[s] = first position of run s.
struct SegFind {
  const u32* keys;
  u32* seg_start;
  u32* seg_of;
  const u32* n_dev;
  u32 cap;
  u32* n_segs_out;
  __device__ u64 size(const Ctl*) const { return min(*n_dev, cap); }
  __device__ u64 value(u64 j) const { return (j == 0 || keys[j] != keys[j - 1]) ? 1u : 0u; }
  __device__ void out(u64 j, u64 excl, u64 v) const {
    if (v && excl < cap) seg_start[excl] = (u32)j;
    if (seg_of) seg_of[j] = (u32)(excl + v - 1);
  }
  __device__ void total(Ctl*, u64 t) const {
    if (t > cap) t = cap;
    *n_segs_out = (u32)t;
    seg_start[t] = (u32)size(nullptr);
  }
};

__device__ __forceinline__ u64 shfl_xor_u64(u64 v, int o) {
  return __shfl_xor_sync(0xFFFFFFFFu, v, o);
}

// Streaming release of leaf-parent entry e, whose child `rel` (its first
// unreleased one) is in this batch's segment [j0, j1): the end r1 of the run
// of present children rel, rel+1, ..., and in *pcs the latest arrival among
// the segment's leaves in that run.  The candidates are the entry's buffered
// leaves (the B entries of its meta vector, all with child >= rel) and the
// segment's leaves; with K of them the first missing child is at most rel+K,
// so a bitmap of K+1 bits, taken from the batch's bitmap scratch, holds the
// whole run.  Returns rel when the scratch is full (ENOSPC).  All 32 lanes
// call it together.
__device__ u32 release_run(const Dev& d, const Batch& b, Ctl* ctl, u32 e, u32 rel, u32 j0, u32 j1,
                           const u32* sperm, u32 n_items, u32* pcs) {
  const int lane = threadIdx.x & 31;
  const int L = d.cfg.depth - 1;
  const u64 n = b.n;
  const u32 B = d.tab.vec_n[2 * (u64)e];
  const u64 K = (u64)B + (j1 - j0);
  const u64 words = (K >> 5) + 1;
  unsigned long long base = 0;
  if (lane == 0) base = atomicAdd((unsigned long long*)&ctl->bm_used, (unsigned long long)words);
  base = __shfl_sync(0xFFFFFFFFu, base, 0);
  if (base + words > d.sc.bm_cap) {
    if (lane == 0) raise_err(ctl, ALTO_ENOSPC);
    *pcs = 0;
    return rel;
  }
  u32* bm = d.sc.bm + base;
  for (u64 w = lane; w < words; w += 32) bm[w] = 0;
  __syncwarp();
  const u64 span = words * 32;
  for (u32 j = j0 + lane; j < j1; j += 32) {
    const u32 x = min(sperm[j], n_items - 1);
    const u32 c = tag_child(b.tags[(u64)L * n + x]);
    if (c >= rel && (u64)(c - rel) < span) atomicOr(&bm[(c - rel) >> 5], 1u << ((c - rel) & 31));
  }
  for (u32 k = lane; k < B; k += 32) {
    bool ok;
    const u64 a = vec_addr(d.tab, e, 0, 2 * (u64)k, &ok);
    if (!ok) continue;
    const u32 c = (u32)d.ar.pool[a];
    if (c >= rel && (u64)(c - rel) < span) atomicOr(&bm[(c - rel) >> 5], 1u << ((c - rel) & 31));
  }
  __syncwarp();
  // first clear bit: K candidates cannot fill K+1 bits, so there is one
  u32 z = kNone;
  for (u64 wb = 0; wb < words && z == kNone; wb += 32) {
    const u64 w = wb + lane;
    u32 cand = kNone;
    if (w < words) {
      const u32 free_bits = ~__ldcg(&bm[w]);
      if (free_bits) cand = (u32)(w * 32) + (u32)(__ffs(free_bits) - 1);
    }
    z = __reduce_min_sync(0xFFFFFFFFu, cand);
  }
  const u32 r1 = (z == kNone) ? rel : rel + z;
  u32 mx = 0;
  for (u32 j = j0 + lane; j < j1; j += 32) {
    const u32 x = min(sperm[j], n_items - 1);
    const u32 c = tag_child(b.tags[(u64)L * n + x]);
    if (c >= rel && c < r1) mx = max(mx, x);
  }
  *pcs = __reduce_max_sync(0xFFFFFFFFu, mx);
  return r1;
}

// Segments longer than this go to k_reduce_big (a block each) instead of a
// warp: a hot group (a million children) would otherwise keep one warp busy
// for the whole batch.
constexpr u32 kBigSeg = 4096;
constexpr int kBigThreads = 512;

// What the reduce of level l reads and writes besides the table.
template <bool LEAF>
struct ReduceArgs {
  int l;
  const u32* skeys;
  const u32* sperm;
  const u32* seg_start;
  const u32* it_rep;
  const u32* it_cseq;
  const u32* it_skey;
  u32* nx_rep;
  u32* nx_cseq;
  u32* nx_skey;
  u32 n_items;
};

template <bool LEAF>
__device__ __forceinline__ ReduceArgs<LEAF> reduce_args(const Dev& d, const Batch& b, int l, const u32* skeys,
                                                         const u32* sperm, const u32* seg_start, int in_set) {
  ReduceArgs<LEAF> r;
  r.l = l;
  r.skeys = skeys;
  r.sperm = sperm;
  r.seg_start = seg_start;
  r.it_rep = d.sc.it_rep[in_set];
  r.it_cseq = d.sc.it_cseq[in_set];
  r.it_skey = d.sc.it_skey[in_set];
  r.nx_rep = d.sc.it_rep[in_set ^ 1];
  r.nx_cseq = d.sc.it_cseq[in_set ^ 1];
  r.nx_skey = d.sc.it_skey[in_set ^ 1];
  r.n_items = LEAF ? b.n : min(d.ctl->n_segs[l + 1], d.cfg.n_max);
  return r;
}

// One item of a segment: a leaf (LEAF) or a child group from the level below.
struct Item {
  u32 rep, done, cs, sk, len, c, last;
};

template <bool LEAF>
__device__ __forceinline__ Item load_item(const Dev& d, const Batch& b, const ReduceArgs<LEAF>& r, u32 j) {
  Item it;
  const u32 x = min(r.sperm[j], r.n_items - 1);
  if (LEAF) {
    it.rep = x;
    it.done = 1;
    it.cs = x;
    it.sk = d.cfg.has_score ? score_key(b.score[x]) : 0u;
    it.len = b.off[x + 1] - b.off[x];
  } else {
    it.rep = r.it_rep[x];
    const u32 cf = r.it_cseq[x];
    it.done = cf >> 31;
    it.cs = cf & 0x7FFFFFFFu;
    it.sk = r.it_skey[x];
    it.len = 0;
  }
  const u64 t = b.tags[(u64)r.l * b.n + it.rep];
  it.c = tag_child(t);
  it.last = tag_last(t);
  return it;
}

// Per-segment reductions over its items.
struct SegRed {
  u32 cnt, m1, fmin, fmax, hasf, cmax, smx, bad, hitrel, below;
  u64 lsum;
  __device__ void init() {
    cnt = m1 = fmax = hasf = cmax = smx = bad = hitrel = below = 0;
    fmin = kNone;
    lsum = 0;
  }
  __device__ void add(const Item& it, u32 rel, bool strm) {
    m1 = max(m1, it.c + 1);
    if (strm) {
      hitrel |= (it.c == rel) ? 1u : 0u;
      below |= (it.c < rel) ? 1u : 0u;
    }
    if (it.last) {
      hasf = 1;
      fmin = min(fmin, it.c);
      fmax = max(fmax, it.c);
    }
    if (it.done) {
      ++cnt;
      cmax = max(cmax, it.cs);
      smx = max(smx, it.sk);
    }
    lsum += it.len;
  }
  __device__ void warp_reduce() {
    cnt = __reduce_add_sync(0xFFFFFFFFu, cnt);
    m1 = __reduce_max_sync(0xFFFFFFFFu, m1);
    fmin = __reduce_min_sync(0xFFFFFFFFu, fmin);
    fmax = __reduce_max_sync(0xFFFFFFFFu, fmax);
    hasf = __reduce_or_sync(0xFFFFFFFFu, hasf);
    cmax = __reduce_max_sync(0xFFFFFFFFu, cmax);
    smx = __reduce_max_sync(0xFFFFFFFFu, smx);
    bad = __reduce_or_sync(0xFFFFFFFFu, bad);
    hitrel = __reduce_or_sync(0xFFFFFFFFu, hitrel);
    below = __reduce_or_sync(0xFFFFFFFFu, below);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) lsum += __shfl_xor_sync(0xFFFFFFFFu, lsum, o);
  }
  __device__ void merge(const SegRed& o) {
    cnt += o.cnt;
    m1 = max(m1, o.m1);
    fmin = min(fmin, o.fmin);
    fmax = max(fmax, o.fmax);
    hasf |= o.hasf;
    cmax = max(cmax, o.cmax);
    smx = max(smx, o.smx);
    bad |= o.bad;
    hitrel |= o.hitrel;
    below |= o.below;
    lsum += o.lsum;
  }
};

// The group's ancestry tags above level l, from its first item; an item
// whose tags differ breaks the ancestry.
struct Chain {
  u64 t[kMaxDepth];
};
__device__ __forceinline__ Chain load_chain(const Batch& b, int l, u32 rep0) {
  Chain h;
#pragma unroll
  for (int q = 0; q < kMaxDepth; ++q) h.t[q] = (q < l) ? b.tags[(u64)q * b.n + rep0] : 0ull;
  return h;
}
__device__ __forceinline__ bool chain_bad(const Batch& b, int l, u32 rep, const Chain& h) {
  bool bad = false;
#pragma unroll
  for (int q = 0; q < kMaxDepth; ++q)
    if (q < l && b.tags[(u64)q * b.n + rep] != h.t[q]) bad = true;
  return bad;
}

// Insert each lane's candidate (0 = none) into the warp's running top-K list
// (lane q holds the q-th best, larger first).  All 32 lanes call it together.
__device__ __forceinline__ void topk_insert(u64& best, u64 cand, int K) {
  const int lane = threadIdx.x & 31;
  const u64 thr = __shfl_sync(0xFFFFFFFFu, best, K - 1);
  u32 pass = __ballot_sync(0xFFFFFFFFu, cand > thr);
  while (pass) {
    const int src = __ffs(pass) - 1;
    pass &= pass - 1;
    const u64 v = __shfl_sync(0xFFFFFFFFu, cand, src);
    const u64 thr2 = __shfl_sync(0xFFFFFFFFu, best, K - 1);
    if (v > thr2) {
      const u32 pos = __popc(__ballot_sync(0xFFFFFFFFu, lane < K && best > v));
      const u64 prev = __shfl_up_sync(0xFFFFFFFFu, best, 1);
      if (lane >= (int)pos && lane < K) best = (lane == (int)pos) ? v : prev;
    }
  }
}

// Streaming release of a segment whose group stays open: the run's end r1,
// and the kept leaves' meta indices and payload offsets (leaves below r1 are
// placed densely straight from the batch; the others are buffered, packed).
// All 32 lanes of one warp call it together.
struct Release {
  u32 r1, pcs, kept_n, kept_len;
};

template <bool LEAF>
__device__ Release stream_release(const Dev& d, const Batch& b, Ctl* ctl, const ReduceArgs<LEAF>& r, u32 e,
                                  u32 rel, u32 j0, u32 j1, const SegRed& red) {
  const int lane = threadIdx.x & 31;
  Release out{rel, 0, 0, 0};
  // the same completion test as the finalize: a group that completes emits its final record instead
  const u32 lo = d.tab.hot[e].last;
  const u32 nl = (lo == kNone && red.hasf) ? red.fmin : lo;
  const bool closes = nl != kNone && d.tab.hot[e].completed + red.cnt == nl + 1 && max(d.tab.hot[e].maxc1, red.m1) <= nl + 1;
  if (closes) return out;
  out.r1 = release_run(d, b, ctl, e, rel, j0, j1, r.sperm, r.n_items, &out.pcs);
  if (out.r1 <= rel) return out;
  for (u32 jb = j0; jb < j1; jb += 32) {
    const u32 j = jb + lane;
    const bool valid = j < j1;
    u32 c = 0, len = 0;
    if (valid) {
      const u32 x = min(r.sperm[j], r.n_items - 1);
      c = tag_child(b.tags[(u64)r.l * b.n + x]);
      len = b.off[x + 1] - b.off[x];
    }
    const bool keep = valid && c >= out.r1;
    const u32 kl = keep ? len : 0u;
    u32 incl = kl;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const u32 y = __shfl_up_sync(0xFFFFFFFFu, incl, o);
      if (lane >= o) incl += y;
    }
    const u32 km = __ballot_sync(0xFFFFFFFFu, keep);
    if (valid) {
      d.sc.leaf_pos[j] = out.kept_len + incl - kl;
      d.sc.leaf_mrank[j] = keep ? out.kept_n + __popc(km & lanemask_lt()) : kNone;
    }
    out.kept_n += __popc(km);
    out.kept_len += __shfl_sync(0xFFFFFFFFu, incl, 31);
  }
  return out;
}

// Merge a reduced segment s of level l into its table entry e: checks,
// completion test, done entry (or a partial release), carry mode, hand-up of
// the concatenation, and the segment's item for level l-1.  One thread.
template <bool LEAF>
__device__ void finalize_segment(const Dev& d, const Batch& b, Ctl* ctl, const ReduceArgs<LEAF>& r, u32 s,
                                 u32 e, u32 rep0, u32 nitems, const SegRed& red, u32 rel, const Release& rl) {
  const int l = r.l;
  const int D = d.cfg.depth;
  const u64 n = b.n;
  const bool carry = LEAF && d.cfg.concat_level >= 0;
  const bool strm = LEAF && d.cfg.stream_leaf;
  if (!LEAF && chain_parent(d.cfg, l)) chain_sync(d.tab, d.ar, ctl, e);
  if (red.bad) raise_err(ctl, ALTO_EINCONSIST);
  if (l > 0 && d.tab.hot[e].up != b.tags[(u64)(l - 1) * n + rep0]) raise_err(ctl, ALTO_EINCONSIST);
  const u32 last_old = d.tab.hot[e].last;
  u32 nl = last_old;
  if (red.hasf) {
    if (red.fmin != red.fmax) raise_err(ctl, ALTO_ELAST);
    if (last_old != kNone && last_old != red.fmin) raise_err(ctl, ALTO_ELAST);
    if (last_old == kNone) nl = red.fmin;
  }
  const u32 m1n = max(d.tab.hot[e].maxc1, red.m1);
  if (nl != kNone && m1n > nl + 1) raise_err(ctl, ALTO_ELAST);
  const u32 comp = d.tab.hot[e].completed + red.cnt;
  const u32 smn = max(d.tab.hot[e].smax, red.smx);
  const bool complete = (nl != kNone) && (comp == nl + 1) && (m1n <= nl + 1);
  d.tab.hot[e].last = nl;
  d.tab.hot[e].maxc1 = m1n;
  d.tab.hot[e].completed = comp;
  d.tab.hot[e].smax = smn;
  const bool part = !complete && rl.r1 > rel;
  // a completing group, or (streaming) a partial release, takes a done entry
  if (complete || part) {
    const u32 cs = part ? rl.pcs : red.cmax;
    u32 di = atomicAdd(&ctl->n_done, 1u);
    if (di < d.sc.done_cap) {
      d.sc.done_e[di] = e;
      d.sc.done_lvl[di] = (u32)l;
      d.sc.done_cseq[di] = cs;
      d.tab.hot[e].done_epoch = ctl->epoch;
      d.tab.done_idx[e] = di;
      if (strm) {
        d.sc.done_part[di] = !part ? 0u : (d.tab.vec_n[2 * (u64)e] ? 2u : 1u);
        d.tab.rnew[e] = part ? rl.r1 : nl + 1;
      }
      if (cs < n) {
        atomicOr(&d.sc.mask[cs], 1u << (D - 1 - l));
        atomicAdd(&d.sc.mblk[cs >> 5], 1u);
      }
    } else {
      raise_err(ctl, ALTO_ENOSPC);
    }
  }
  if (carry) {
    // 1: to the arena, 2: placed densely, 3: a partial release, both
    d.sc.seg_carry[s] = complete ? 2u : (part ? 3u : 1u);
    if (!complete) {
      const u32 v0 = d.tab.vec_n[2 * (u64)e], v1 = d.tab.vec_n[2 * (u64)e + 1];
      d.sc.seg_vb0[s] = v0;
      d.sc.seg_vb1[s] = v1;
      d.tab.vec_n[2 * (u64)e] = v0 + (part ? rl.kept_n : nitems);
      d.tab.vec_n[2 * (u64)e + 1] = v1 + (part ? rl.kept_len : (u32)red.lsum);
    }
  }
  if (chain_level(d.cfg, l) && complete) {
    const u64 tp = b.tags[(u64)(l - 1) * n + rep0];
    const u64 upp = (l > 1) ? b.tags[(u64)(l - 2) * n + rep0] : 0ull;
    int ins = 0;
    const u32 P = ht_find_or_insert(d.tab, ((u64)(l - 1) << 32) | tag_pid(tp), upp, ctl, &ins, b.tags, n,
                                    rep0, l - 1);
    if (ins) atomicAdd((unsigned long long*)&ctl->live_groups, 1ull);
    const u64 total = (u64)d.tab.vec_n[2 * (u64)e + 1] + (LEAF ? red.lsum : 0ull);
    if (P != kNone) chain_reserve(d.tab, e, P, tag_child(tp), total);
  }
  if (l > 0) {
    r.nx_rep[s] = rep0;
    r.nx_cseq[s] = (complete ? 0x80000000u : 0u) | red.cmax;
    r.nx_skey[s] = smn;
  }
}

// Segments of at most kSmallSeg items are reduced by eight lanes (a warp takes
// four at a time): most groups have a few dozen children or fewer, and a
// whole warp per group left most lanes idle.
constexpr u32 kSmallSeg = 32;

// A small segment [j0, j1) by the eight lanes of `gmask` (sub = lane index in
// the group): up to four items a lane, all loaded before they are combined;
// the top-k of a TOPK level merged by the group's first lane.
template <bool LEAF>
__device__ __forceinline__ void reduce_small(const Dev& d, const Batch& b, Ctl* ctl, const ReduceArgs<LEAF>& r,
                                             u32 s, u32 j0, u32 j1, u32 gmask, int sub, bool topk, int K) {
  const u32 e = r.skeys[j0] & d.tab.mask;
  const u32 rep0 = LEAF ? min(r.sperm[j0], r.n_items - 1) : r.it_rep[min(r.sperm[j0], r.n_items - 1)];
  const bool strm = LEAF && d.cfg.stream_leaf;
  const u32 rel = strm ? d.tab.rel[e] : 0u;
  const Chain htag = load_chain(b, r.l, rep0);
  SegRed red;
  red.init();
  u64 cand[kSmallSeg / 8];
  u32 len[kSmallSeg / 8];
#pragma unroll
  for (int q = 0; q < (int)(kSmallSeg / 8); ++q) {
    const u32 j = j0 + 8 * q + sub;
    cand[q] = 0;
    len[q] = 0;
    if (j < j1) {
      const Item it = load_item<LEAF>(d, b, r, j);
      red.add(it, rel, strm);
      if (chain_bad(b, r.l, it.rep, htag)) red.bad = 1;
      len[q] = it.len;
      if (it.done) cand[q] = ((u64)it.sk << 32) | (u64)(~it.c);
    }
  }
  if (LEAF) {
    // payload offset of each leaf inside the segment
    u32 running = 0;
#pragma unroll
    for (int q = 0; q < (int)(kSmallSeg / 8); ++q) {
      u32 incl = len[q];
#pragma unroll
      for (int o = 1; o < 8; o <<= 1) {
        const u32 y = __shfl_up_sync(gmask, incl, o, 8);
        if (sub >= o) incl += y;
      }
      const u32 j = j0 + 8 * q + sub;
      if (j < j1) d.sc.leaf_pos[j] = running + incl - len[q];
      running += __shfl_sync(gmask, incl, 7, 8);
    }
  }
  red.cnt = __reduce_add_sync(gmask, red.cnt);
  red.m1 = __reduce_max_sync(gmask, red.m1);
  red.fmin = __reduce_min_sync(gmask, red.fmin);
  red.fmax = __reduce_max_sync(gmask, red.fmax);
  red.hasf = __reduce_or_sync(gmask, red.hasf);
  red.cmax = __reduce_max_sync(gmask, red.cmax);
  red.smx = __reduce_max_sync(gmask, red.smx);
  red.bad = __reduce_or_sync(gmask, red.bad);
#pragma unroll
  for (int o = 4; o > 0; o >>= 1) red.lsum += __shfl_xor_sync(gmask, red.lsum, o, 8);
  if (strm) {
    // a group that stays open and whose first unreleased child came releases
    // a run: that needs a whole warp, so the segment is left to k_reduce_rel
    red.hitrel = __reduce_or_sync(gmask, red.hitrel);
    red.below = __reduce_or_sync(gmask, red.below);
    if (red.below && sub == 0) raise_err(ctl, ALTO_EDUP);
    if (red.hitrel) {
      const u32 lo = d.tab.hot[e].last;
      const u32 nl = (lo == kNone && red.hasf) ? red.fmin : lo;
      const bool closes = nl != kNone && d.tab.hot[e].completed + red.cnt == nl + 1 &&
                          max(d.tab.hot[e].maxc1, red.m1) <= nl + 1;
      if (!closes) {
        if (sub == 0) {
          const u32 q = atomicAdd(&ctl->n_rel, 1u);
          if (q < d.cfg.n_max) d.sc.rel_seg[q] = s;
          else raise_err(ctl, ALTO_ENOSPC);
        }
        return;
      }
    }
  }
  if (topk) {
    // the group's first lane keeps the list, best first, in local memory
    u64 list[kMaxTopk];
    int have = 0;
    if (sub == 0) {
      have = (int)min(d.tab.hot[e].completed, (u32)K);
      for (int i = 0; i < have; ++i) list[i] = d.tab.topk[(u64)e * d.tab.kk + i];
    }
#pragma unroll
    for (int q = 0; q < (int)(kSmallSeg / 8); ++q) {
      for (int t = 0; t < 8; ++t) {
        const u64 v = __shfl_sync(gmask, cand[q], t, 8);
        if (sub != 0 || v == 0) continue;
        if (have == K && v <= list[K - 1]) continue;
        int pos = have < K ? have : K - 1;
        while (pos > 0 && list[pos - 1] < v) {
          list[pos] = list[pos - 1];
          --pos;
        }
        list[pos] = v;
        if (have < K) ++have;
      }
    }
    if (sub == 0)
      for (int i = 0; i < K; ++i) d.tab.topk[(u64)e * d.tab.kk + i] = (i < have) ? list[i] : 0ull;
  }
  if (sub == 0) finalize_segment<LEAF>(d, b, ctl, r, s, e, rep0, j1 - j0, red, 0u, Release{0, 0, 0, 0});
}

// A segment by the whole warp (32 lanes).
template <bool LEAF>
__device__ __forceinline__ void reduce_warp(const Dev& d, const Batch& b, Ctl* ctl, const ReduceArgs<LEAF>& r,
                                            u32 s, u32 j0, u32 j1, bool topk, int K, bool strm) {
  const int lane = threadIdx.x & 31;
  const u32 e = r.skeys[j0] & d.tab.mask;
  const u32 rep0 = LEAF ? min(r.sperm[j0], r.n_items - 1) : r.it_rep[min(r.sperm[j0], r.n_items - 1)];
  const u32 rel = strm ? d.tab.rel[e] : 0u;
  const Chain htag = load_chain(b, r.l, rep0);
  SegRed red;
  red.init();
  u32 running = 0;  // payload elements of the segment's earlier leaves (leaf level)
  for (u32 jb = j0; jb < j1; jb += 32) {
    const u32 j = jb + lane;
    const bool valid = j < j1;
    u32 len = 0;
    if (valid) {
      const Item it = load_item<LEAF>(d, b, r, j);
      red.add(it, rel, strm);
      if (chain_bad(b, r.l, it.rep, htag)) red.bad = 1;
      len = it.len;
    }
    if (LEAF) {
      u32 incl = len;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const u32 y = __shfl_up_sync(0xFFFFFFFFu, incl, o);
        if (lane >= o) incl += y;
      }
      if (valid) d.sc.leaf_pos[j] = running + incl - len;
      running += __shfl_sync(0xFFFFFFFFu, incl, 31);
    }
  }
  red.warp_reduce();
  Release rl{rel, 0, 0, 0};
  if (strm) {
    if (red.below && lane == 0) raise_err(ctl, ALTO_EDUP);
    if (red.hitrel) rl = stream_release<LEAF>(d, b, ctl, r, e, rel, j0, j1, red);
    __syncwarp();
  }
  if (topk) {
    // running top-k of complete children: lane q holds the q-th best
    const u32 valid = min(d.tab.hot[e].completed, (u32)K);
    u64 best = (lane < (int)valid) ? d.tab.topk[(u64)e * d.tab.kk + lane] : 0ull;
    for (u32 jb = j0; jb < j1; jb += 32) {
      const u32 j = jb + lane;
      u64 cand = 0;
      if (j < j1) {
        const Item it = load_item<LEAF>(d, b, r, j);
        if (it.done) cand = ((u64)it.sk << 32) | (u64)(~it.c);
      }
      topk_insert(best, cand, K);
    }
    if (lane < K) d.tab.topk[(u64)e * d.tab.kk + lane] = best;
  }
  if (lane == 0) finalize_segment<LEAF>(d, b, ctl, r, s, e, rep0, j1 - j0, red, rel, rl);
}

// The groups present at level l: reduce their items, merge with the table
// entries, test completion, and emit each group as an item of level l-1.  A
// warp takes four segments at a time: the small ones by eight lanes each,
// the others one after another by the whole warp; segments longer than
// kBigSeg are listed for k_reduce_big.  (A small segment whose group makes a
// streaming release is listed for k_reduce_rel: the release needs a warp.)
template <bool LEAF, bool G>
__global__ void __launch_bounds__(kThreads) k_reduce(Dev d, Batch bv, int l, const u32* skeys,
                                                     const u32* sperm, const u32* seg_start,
                                                     int in_set) {
  pdl_enter();
  const Batch b = batch_of<G>(bv, d);
  Ctl* ctl = d.ctl;
  if (poisoned(ctl)) return;
  const u32 nseg = min(ctl->n_segs[l], d.cfg.n_max);
  const int lane = threadIdx.x & 31, grp = lane >> 3, sub = lane & 7;
  const u32 gmask = 0xFFu << (8 * grp);
  const u32 gw = gtid() >> 5, nw = gstride() >> 5;
  const bool topk = d.cfg.score_op[l] == ALTO_SCORE_TOPK;
  const int K = d.cfg.topk_k[l];
  const bool strm = LEAF && d.cfg.stream_leaf;
  const ReduceArgs<LEAF> r = reduce_args<LEAF>(d, b, l, skeys, sperm, seg_start, in_set);
  for (u32 sb = gw * 4; sb < nseg; sb += nw * 4) {
    const u32 s = sb + grp;
    u32 j0 = 0, j1 = 0;
    if (s < nseg) {
      j1 = min(seg_start[s + 1], r.n_items);
      j0 = min(seg_start[s], j1);
    }
    const bool small = j1 > j0 && j1 - j0 <= kSmallSeg;
    if (small) reduce_small<LEAF>(d, b, ctl, r, s, j0, j1, gmask, sub, topk, K);
    u32 rest = __ballot_sync(0xFFFFFFFFu, sub == 0 && j1 > j0 && !small);
    while (rest) {
      const int g = (__ffs(rest) - 1) >> 3;
      rest &= rest - 1;
      const u32 s2 = sb + g;
      const u32 a0 = __shfl_sync(0xFFFFFFFFu, j0, 8 * g), a1 = __shfl_sync(0xFFFFFFFFu, j1, 8 * g);
      if (a1 - a0 > kBigSeg) {
        if (lane == 0) {
          const u32 q = atomicAdd(&ctl->n_big[l], 1u);
          if (q < d.sc.big_cap) d.sc.big_seg[(u64)l * d.sc.big_cap + q] = s2;
          else raise_err(ctl, ALTO_ENOSPC);
        }
        continue;
      }
      reduce_warp<LEAF>(d, b, ctl, r, s2, a0, a1, topk, K, strm);
    }
  }
}

// Streaming release: the small segments whose groups release a run, a warp each.
template <bool G>
__global__ void __launch_bounds__(kThreads) k_reduce_rel(Dev d, Batch bv, const u32* skeys, const u32* sperm,
                                                         const u32* seg_start, int in_set) {
  pdl_enter();
  const Batch b = batch_of<G>(bv, d);
  Ctl* ctl = d.ctl;
  if (poisoned(ctl)) return;
  const int l = d.cfg.depth - 1;
  const u32 nrel = min(ctl->n_rel, d.cfg.n_max);
  const u32 gw = gtid() >> 5, nw = gstride() >> 5;
  const bool topk = d.cfg.score_op[l] == ALTO_SCORE_TOPK;
  const int K = d.cfg.topk_k[l];
  const ReduceArgs<true> r = reduce_args<true>(d, b, l, skeys, sperm, seg_start, in_set);
  for (u32 q = gw; q < nrel; q += nw) {
    const u32 s = d.sc.rel_seg[q];
    const u32 j1 = min(seg_start[s + 1], r.n_items);
    const u32 j0 = min(seg_start[s], j1);
    if (j0 < j1) reduce_warp<true>(d, b, ctl, r, s, j0, j1, topk, K, true);
  }
}

// The segments longer than kBigSeg, a block of kBigThreads each: the same
// reductions with the block's warps over strided items, combined in shared
// memory; each warp keeps a top-k of its items and warp 0 merges them with
// the entry's list; a streaming release runs on warp 0.
template <bool LEAF, bool G>
__global__ void __launch_bounds__(kBigThreads) k_reduce_big(Dev d, Batch bv, int l, const u32* skeys,
                                                            const u32* sperm, const u32* seg_start,
                                                            int in_set) {
  pdl_enter();
  const Batch b = batch_of<G>(bv, d);
  Ctl* ctl = d.ctl;
  if (poisoned(ctl)) return;
  constexpr int kW = kBigThreads / 32;
  __shared__ SegRed s_red[kW];
  __shared__ u64 s_topk[kW][kMaxTopk];
  __shared__ u32 s_scan[kW];
  const u32 nbig = min(ctl->n_big[l], d.sc.big_cap);
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const bool topk = d.cfg.score_op[l] == ALTO_SCORE_TOPK;
  const int K = d.cfg.topk_k[l];
  const bool strm = LEAF && d.cfg.stream_leaf;
  const ReduceArgs<LEAF> r = reduce_args<LEAF>(d, b, l, skeys, sperm, seg_start, in_set);
  for (u32 q = blockIdx.x; q < nbig; q += gridDim.x) {
    const u32 s = d.sc.big_seg[(u64)l * d.sc.big_cap + q];
    const u32 j1 = min(seg_start[s + 1], r.n_items);
    const u32 j0 = min(seg_start[s], j1);
    const u32 e = skeys[j0] & d.tab.mask;
    const u32 rep0 = LEAF ? min(sperm[j0], r.n_items - 1) : r.it_rep[min(sperm[j0], r.n_items - 1)];
    const u32 rel = strm ? d.tab.rel[e] : 0u;
    const Chain htag = load_chain(b, l, rep0);
    SegRed red;
    red.init();
    u64 best = 0;
    u32 running = 0;
    // items in block-wide steps: reductions, the leaves' payload offsets
    // (a block scan per step), and each warp's top-k
    for (u32 jb = j0; jb < j1; jb += kBigThreads) {
      const u32 j = jb + threadIdx.x;
      const bool valid = j < j1;
      u32 len = 0;
      u64 cand = 0;
      if (valid) {
        const Item it = load_item<LEAF>(d, b, r, j);
        red.add(it, rel, strm);
        if (chain_bad(b, l, it.rep, htag)) red.bad = 1;
        len = it.len;
        if (it.done) cand = ((u64)it.sk << 32) | (u64)(~it.c);
      }
      if (topk) topk_insert(best, cand, K);
      if (LEAF) {
        u32 incl = len;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
          const u32 y = __shfl_up_sync(0xFFFFFFFFu, incl, o);
          if (lane >= o) incl += y;
        }
        if (lane == 31) s_scan[warp] = incl;
        __syncthreads();
        u32 wbase = 0, total = 0;
        for (int w = 0; w < kW; ++w) {
          const u32 v = s_scan[w];
          if (w < warp) wbase += v;
          total += v;
        }
        if (valid) d.sc.leaf_pos[j] = running + wbase + incl - len;
        running += total;
        __syncthreads();
      }
    }
    red.warp_reduce();
    if (lane == 0) s_red[warp] = red;
    if (topk && lane < K) s_topk[warp][lane] = best;
    __syncthreads();
    if (warp == 0) {
      SegRed all = s_red[0];
      for (int w = 1; w < kW; ++w) all.merge(s_red[w]);
      Release rl{rel, 0, 0, 0};
      if (strm) {
        if (all.below && lane == 0) raise_err(ctl, ALTO_EDUP);
        if (all.hitrel) rl = stream_release<LEAF>(d, b, ctl, r, e, rel, j0, j1, all);
        __syncwarp();
      }
      if (topk) {
        const u32 valid = min(d.tab.hot[e].completed, (u32)K);
        u64 bt = (lane < (int)valid) ? d.tab.topk[(u64)e * d.tab.kk + lane] : 0ull;
        for (int w = 0; w < kW; ++w) topk_insert(bt, (lane < K) ? s_topk[w][lane] : 0ull, K);
        if (lane < K) d.tab.topk[(u64)e * d.tab.kk + lane] = bt;
      }
      if (lane == 0) finalize_segment<LEAF>(d, b, ctl, r, s, e, rep0, j1 - j0, all, rel, rl);
    }
    __syncthreads();
  }
}

// ---------------------------------------------------------------------------
// upper levels without TOPK: hash-table entries accumulate the batch's items
// with warp-aggregated atomics; the touched entries are then finalised.
// ---------------------------------------------------------------------------
// One item of level l per lane (all 32 lanes together; `valid` marks the
// real ones): the batch's first item of an entry puts the entry on the
// level's touched list, and every item adds itself to the entry's batch
// accumulators, warp-aggregated over lanes with the same entry.
__device__ __forceinline__ void add_items(const Dev& d, Ctl* ctl, bool valid, u32 e, u32 rep, u32 c, u32 f,
                                          u32 done, u32 cs, u32 sk, u32 ep, u32* list, u32* list_n,
                                          BlockTake* bsh = nullptr) {
  bool first = false;
  if (valid) first = atomicExch(&d.tab.hot[e].touch, ep) != ep;
  {
    // (with `bsh`, all threads of the block call this together)
    const u32 pos = bsh ? block_take(first, list_n, *bsh) : warp_take(first, list_n);
    if (first) {
      if (pos < d.cfg.n_max) list[pos] = e;
      d.tab.hot[e].acc_rep = rep;
    }
  }
  // lanes without an item form their own group; the whole warp takes part
  const u32 key = valid ? e : kNone;
  const u32 peers = __match_any_sync(0xFFFFFFFFu, key);
  if (__all_sync(0xFFFFFFFFu, peers == (1u << (threadIdx.x & 31)))) {
    if (valid) {
      if (done) {
        atomicAdd((unsigned long long*)&d.tab.hot[e].acc_cl, 1ull << 40);
        atomicMax(&d.tab.hot[e].acc_cs1, cs + 1);
        if (sk) atomicMax(&d.tab.hot[e].acc_smx, sk);
      }
      atomicMax(&d.tab.hot[e].acc_m1, c + 1);
      if (f) {
        atomicMin(&d.tab.hot[e].acc_fmin, c);
        atomicMax(&d.tab.hot[e].acc_fmax1, c + 1);
      }
    }
    return;
  }
  const int leader = __ffs(peers) - 1;
  const u32 cnt = __reduce_add_sync(peers, done);
  const u32 m1 = __reduce_max_sync(peers, valid ? c + 1 : 0u);
  const u32 fmin = __reduce_min_sync(peers, (valid && f) ? c : kNone);
  const u32 fmax1 = __reduce_max_sync(peers, (valid && f) ? c + 1 : 0u);
  const u32 cs1 = __reduce_max_sync(peers, (valid && done) ? cs + 1 : 0u);
  const u32 smx = __reduce_max_sync(peers, (valid && done) ? sk : 0u);
  if (valid && (int)(threadIdx.x & 31) == leader) {
    if (cnt) atomicAdd((unsigned long long*)&d.tab.hot[e].acc_cl, (unsigned long long)cnt << 40);
    if (m1) atomicMax(&d.tab.hot[e].acc_m1, m1);
    if (fmin != kNone) atomicMin(&d.tab.hot[e].acc_fmin, fmin);
    if (fmax1) atomicMax(&d.tab.hot[e].acc_fmax1, fmax1);
    if (cs1) atomicMax(&d.tab.hot[e].acc_cs1, cs1);
    if (smx) atomicMax(&d.tab.hot[e].acc_smx, smx);
  }
}

// Ancestry of item `rep` (tags 0..l-1) against entry e's chain row, which the
// entry's inserter may be writing in this same launch: wait (bounded) until
// it says the row is written, then read the row from L2 (an L1 line of this
// SM may predate the write).
__device__ bool chain_differs_ready(const Dev& d, Ctl* ctl, u32 e, const Batch& b, u32 rep, int l) {
  if (l == 0) return false;  // a top-level group has no ancestry to compare
  u64 spins = 0;
  for (;;) {
    u32 r;
    asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(r) : "l"(d.tab.ready + e) : "memory");
    if (r) break;
    if (*(volatile int*)&ctl->abort) return false;
    if (++spins > d.cfg.spin_limit) {
      raise_timeout(ctl);
      return false;
    }
    __nanosleep(32);
  }
  const ulonglong2* row = reinterpret_cast<const ulonglong2*>(d.tab.chain + (u64)e * d.tab.chain_len);
  bool bad = false;
  for (int q = 0; q < l; q += 2) {
    const ulonglong2 v = __ldcg(row + (q >> 1));
    if (b.tags[(u64)q * b.n + rep] != v.x) bad = true;
    if (q + 1 < l && b.tags[(u64)(q + 1) * b.n + rep] != v.y) bad = true;
  }
  return bad;
}

// Items of level l (after a TOPK level or the sorted leaf level, whose
// reduce does not look up parents): check ancestry against the entry and
// accumulate; the touched entries go to `list`.
template <bool G>
__global__ void __launch_bounds__(kThreads) k_up_accumulate(Dev d, Batch bv, int l, int in_set, u32* list) {
  pdl_enter();
  const Batch b = batch_of<G>(bv, d);
  Ctl* ctl = d.ctl;
  if (poisoned(ctl)) return;
  const u32 ni = min(ctl->n_segs[l + 1], d.cfg.n_max);
  const u32 ep = ctl->epoch;
  const u32* it_rep = d.sc.it_rep[in_set];
  const u32* it_cseq = d.sc.it_cseq[in_set];
  const u32* it_skey = d.sc.it_skey[in_set];
  const u64 n = b.n;
  const u32 end = (ni + 31) & ~31u;
  for (u32 x = gtid(); x < end; x += gstride()) {
    const bool valid = x < ni;
    u32 e = 0, rep = 0, c = 0, f = 0, done = 0, cs = 0, sk = 0;
    if (valid) {
      e = d.sc.up_sort_keys0[x] & d.tab.mask;
      rep = it_rep[x];
      const u64 t = b.tags[(u64)l * n + rep];
      c = tag_child(t);
      f = tag_last(t);
      const u32 cf = it_cseq[x];
      done = cf >> 31;
      cs = cf & 0x7FFFFFFFu;
      sk = it_skey[x];
      if (chain_differs(d.tab, e, b.tags, n, rep, l)) raise_err(ctl, ALTO_EINCONSIST);
    }
    add_items(d, ctl, valid, e, rep, c, f, done, cs, sk, ep, list, &ctl->n_segs[l]);
  }
}

// Leaf level without TOPK: every fragment, in arrival order (coalesced),
// checks its ancestry against its group's entry and adds itself to the
// entry's batch accumulators (warp-aggregated over lanes of the same group).
// 32 registers: eight blocks per SM, so the grid is one wave
template <bool G>
__global__ void __launch_bounds__(kThreads, 8) k_leaf_accumulate(Dev d, Batch bv) {
  pdl_enter();
  const Batch b = batch_of<G>(bv, d);
  Ctl* ctl = d.ctl;
  if (poisoned(ctl)) return;
  __shared__ u32 s_cnt, s_base;
  if (threadIdx.x == 0) s_cnt = 0;
  __syncthreads();
  const int D = d.cfg.depth;
  const int L = D - 1;
  const u64 n = b.n;
  const bool scores = d.cfg.has_score;
  const u32 ep7 = epoch7(ctl);
  u32* list = d.sc.leaf_seg_start;  // touched leaf-parent entries
  // whole blocks iterate together: the touched entries are appended to the
  // list with one atomic per block and round
  const u32 end = (b.n + kThreads - 1) / kThreads * kThreads;
  const int lane = threadIdx.x & 31;
  for (u32 i = gtid(); i < end; i += gstride()) {
    const bool valid = i < b.n;
    u32 e = 0, c = 0, f = 0, len = 0, sk = 0;
    if (valid) {
      e = d.sc.leaf_sort_keys0[i] & d.tab.mask;
      const u64 t = b.tags[(u64)L * n + i];
      c = tag_child(t);
      f = tag_last(t);
      len = b.off[i + 1] - b.off[i];
      if (scores) sk = score_key(b.score[i]);
    }
    const u32 key = valid ? e : kNone;
    const u32 peers = __match_any_sync(0xFFFFFFFFu, key);
    // The accumulator atomics, the chain row loads and the leaf-slot probe
    // depend on the entry only: all of them go out before any result is used.
    bool first = false;  // this lane made the entry's first contribution of the batch
    bool bad = false, dup = false;
    if (__all_sync(0xFFFFFFFFu, peers == (1u << lane))) {
      // every lane its own group (the common case): plain atomics, no reductions
      if (valid) {
        Hot* rec = d.tab.hot + e;
        const u64 old = atomicAdd((unsigned long long*)&rec->acc_cl, (1ull << 40) | len);
        atomicMax(&rec->acc_m1, c + 1);
        atomicMax(&rec->acc_cs1, i + 1);
        if (f) {
          atomicMin(&rec->acc_fmin, c);
          atomicMax(&rec->acc_fmax1, c + 1);
        }
        if (scores) atomicMax(&rec->acc_smx, sk);
        bad = chain_differs(d.tab, e, b.tags, n, i, L);
        dup = leaf_dup(d.tab, d.sc, e, c, ep7, ctl);
        first = old == 0;
      }
    } else {
      const int leader = __ffs(peers) - 1;
      const u32 cnt = __popc(peers);
      const u32 m1 = __reduce_max_sync(peers, valid ? c + 1 : 0u);
      const u32 cs1 = __reduce_max_sync(peers, valid ? i + 1 : 0u);
      const u32 lsum = __reduce_add_sync(peers, len);
      const u32 anyf = __reduce_or_sync(peers, f);
      const u32 fmin = anyf ? __reduce_min_sync(peers, (valid && f) ? c : kNone) : kNone;
      const u32 fmax1 = anyf ? __reduce_max_sync(peers, (valid && f) ? c + 1 : 0u) : 0u;
      const u32 smx = scores ? __reduce_max_sync(peers, valid ? sk : 0u) : 0u;
      u64 old = 1;
      if (valid && lane == leader) {
        // one returning atomic per group and warp: leaves and payload together
        Hot* rec = d.tab.hot + e;
        old = atomicAdd((unsigned long long*)&rec->acc_cl, ((unsigned long long)cnt << 40) | lsum);
        atomicMax(&rec->acc_m1, m1);
        atomicMax(&rec->acc_cs1, cs1);
        if (fmax1) {
          atomicMin(&rec->acc_fmin, fmin);
          atomicMax(&rec->acc_fmax1, fmax1);
        }
        if (smx) atomicMax(&rec->acc_smx, smx);
      }
      if (valid) {
        bad = chain_differs(d.tab, e, b.tags, n, i, L);
        dup = leaf_dup(d.tab, d.sc, e, c, ep7, ctl);
      }
      first = old == 0;
    }
    if (bad) raise_err(ctl, ALTO_EINCONSIST);
    if (dup) raise_err(ctl, ALTO_EDUP);
    const u32 m = __ballot_sync(0xFFFFFFFFu, first);
    const int wl = __ffs(m) - 1;
    u32 wbase = 0;
    if (m != 0 && lane == wl) wbase = atomicAdd(&s_cnt, (u32)__popc(m));
    __syncthreads();
    if (threadIdx.x == 0) {
      s_base = s_cnt ? atomicAdd(&ctl->n_segs[L], s_cnt) : 0u;
      s_cnt = 0;
    }
    __syncthreads();
    if (m != 0) wbase = __shfl_sync(0xFFFFFFFFu, wbase, wl);
    if (first) {
      const u32 pos = s_base + wbase + __popc(m & lanemask_lt());
      if (pos < d.cfg.n_max) list[pos] = e;
      d.tab.hot[e].acc_rep = i;
    }
  }
}

// One thread per touched entry: merge, test completion, emit the next items.
template <bool LEAF, bool G>
__global__ void __launch_bounds__(kThreads) k_up_finalize(Dev d, Batch bv, int l, int in_set,
                                                          const u32* list, u32* list_next) {
  pdl_enter();
  const Batch b = batch_of<G>(bv, d);
  Ctl* ctl = d.ctl;
  if (poisoned(ctl)) return;
  const int D = d.cfg.depth;
  const bool carry = LEAF && d.cfg.concat_level >= 0;
  const bool receives = !LEAF && chain_parent(d.cfg, l);
  const bool hands_up = chain_level(d.cfg, l);
  // the level above takes its items right here (no separate accumulate
  // launch) unless it is a TOPK level, whose items are sorted instead
  const bool merge = l > 0 && d.cfg.score_op[l - 1] != ALTO_SCORE_TOPK;
  const u32 nt = min(ctl->n_segs[l], d.cfg.n_max);
  const u32 ep = ctl->epoch;
  const u32 ep7 = epoch7(ctl);
  // appends to the done and touched lists and the chunk allocation take one
  // atomic per block on their shared counters
  __shared__ u32 s_ins;
  __shared__ BlockTake s_done, s_list;
  __shared__ GrowShared s_grow;
  if (threadIdx.x == 0) {
    s_ins = 0;
    s_done.cnt = 0;
    s_list.cnt = 0;
    s_grow.got = 0;
  }
  if (threadIdx.x < kNumChunks) {
    s_grow.cnt[threadIdx.x] = 0;
    s_grow.rank[threadIdx.x] = 0;
  }
  __syncthreads();
  u32* nx_rep = d.sc.it_rep[in_set ^ 1];
  u32* nx_cseq = d.sc.it_cseq[in_set ^ 1];
  u32* nx_skey = d.sc.it_skey[in_set ^ 1];
  const u64 n = b.n;
  const u32 end = (nt + kThreads - 1) / kThreads * kThreads;  // whole blocks iterate together
  for (u32 s = gtid(); s < end; s += gstride()) {
    const bool valid = s < nt;
    u32 e = 0, rep = 0, cmax = 0, smn = 0, blen = 0;
    bool complete = false, grows = false;
    u64 gv[4] = {0, 0, 0, 0};  // old and new element counts of the two arena vectors
    if (valid) {
      e = list[s] & d.tab.mask;
      if (receives) chain_sync(d.tab, d.ar, ctl, e);
      // the entry's record in four 16-byte loads; the accumulators are reset
      // for the next batch with two stores
      uint4* hw = reinterpret_cast<uint4*>(d.tab.hot + e);
      const uint4 h0 = hw[0], a = hw[1], f = hw[2], h3 = hw[3];
      const u64 cl = ((u64)a.y << 32) | a.x;
      const u32 cnt = (u32)(cl >> 40), m1 = a.z, cs1 = a.w;
      if (LEAF) blen = (u32)(cl & kPos40);
      const u32 fmin = f.x, fmax1 = f.y, smx = f.z;
      rep = f.w;
      hw[1] = make_uint4(0, 0, 0, 0);
      hw[2] = make_uint4(kNone, 0, 0, 0);
      const u64 up_e = ((u64)h0.y << 32) | h0.x;
      if (l > 0 && up_e != b.tags[(u64)(l - 1) * n + rep]) raise_err(ctl, ALTO_EINCONSIST);
      const u32 last_old = h0.z;
      u32 nl = last_old;
      if (fmax1) {
        if (fmin + 1 != fmax1) raise_err(ctl, ALTO_ELAST);
        if (last_old != kNone && last_old != fmin) raise_err(ctl, ALTO_ELAST);
        if (last_old == kNone) nl = fmin;
      }
      const u32 m1n = max(h3.x, m1);
      if (nl != kNone && m1n > nl + 1) raise_err(ctl, ALTO_ELAST);
      const u32 comp = h0.w + cnt;
      smn = max(h3.y, smx);
      complete = (nl != kNone) && (comp == nl + 1) && (m1n <= nl + 1);
      d.tab.hot[e].last = nl;
      d.tab.hot[e].maxc1 = m1n;
      d.tab.hot[e].completed = comp;
      d.tab.hot[e].smax = smn;
      cmax = cs1 ? cs1 - 1 : 0;
      if (carry && !complete) {
        // reserve this batch's leaves at the end of the group's arena vectors
        const u32 v0 = d.tab.vec_n[2 * (u64)e], v1 = d.tab.vec_n[2 * (u64)e + 1];
        d.tab.cur[e] = ((u64)v0 << 40) | v1;
        d.tab.vec_n[2 * (u64)e] = v0 + cnt;
        d.tab.vec_n[2 * (u64)e + 1] = v1 + blen;
        d.tab.bstate[e] = make_uint4(ep, 1u, 0u, 0u);
        grows = true;
        gv[0] = 2 * (u64)v0;
        gv[1] = 2 * ((u64)v0 + cnt);
        gv[2] = v1;
        gv[3] = (u64)v1 + blen;
      }
    }
    // the leaf level allocates the chunks of the reserved growth right here
    if (LEAF && carry) block_grow(d.tab, d.ar, ctl, grows, e, gv[0], gv[1], gv[2], gv[3], s_grow);
    const u32 di = block_take(complete, &ctl->n_done, s_done);
    if (valid && complete) {
      if (di < d.sc.done_cap) {
        d.sc.done_e[di] = e;
        d.sc.done_lvl[di] = (u32)l;
        d.sc.done_cseq[di] = cmax;
        d.tab.hot[e].done_epoch = ep;
        d.tab.done_idx[e] = di;
        if (cmax < n) {
          atomicOr(&d.sc.mask[cmax], 1u << (D - 1 - l));
          atomicAdd(&d.sc.mblk[cmax >> 5], 1u);
          // split placement: leaf parents are ranked among themselves
          if (LEAF && d.split) atomicAdd(&d.sc.lblk[cmax >> 5], 1u);
        }
      } else {
        raise_err(ctl, ALTO_ENOSPC);
      }
    }
    if (l > 0) {
      u32 e2 = kNone, c2 = 0, f2 = 0;
      if (valid) {
        if (!merge) {
          nx_rep[s] = rep;
          nx_cseq[s] = (complete ? 0x80000000u : 0u) | cmax;
          nx_skey[s] = smn;
        }
        // the next level's item is known now: find or insert its parent group
        const u64 tp = b.tags[(u64)(l - 1) * n + rep];
        const u64 upp = (l > 1) ? b.tags[(u64)(l - 2) * n + rep] : 0ull;
        int ins = 0;
        e2 = ht_find_or_insert(d.tab, ((u64)(l - 1) << 32) | tag_pid(tp), upp, ctl, &ins, b.tags, n, rep,
                               l - 1, merge);
        if (ins) atomicAdd(&s_ins, 1u);
        if (!merge) d.sc.up_sort_keys0[s] = (e2 == kNone) ? 0u : e2;
        if (e2 != kNone) {
          c2 = tag_child(tp);
          f2 = tag_last(tp);
          if (ps_insert(d.sc, e2, c2, ep7, ctl)) raise_err(ctl, ALTO_EINCONSIST);
          if (hands_up && complete) chain_reserve(d.tab, e, e2, c2, (u64)d.tab.vec_n[2 * (u64)e + 1] + blen);
          // an inserter wrote the row from this very fragment's tags
          if (merge && !ins && chain_differs_ready(d, ctl, e2, b, rep, l - 1)) raise_err(ctl, ALTO_EINCONSIST);
        }
      }
      if (merge)
        add_items(d, ctl, e2 != kNone, e2, rep, c2, f2, complete ? 1u : 0u, cmax, smn, ep, list_next,
                  &ctl->n_segs[l - 1], &s_list);
    }
  }
  __syncthreads();
  if (threadIdx.x == 0 && s_ins) atomicAdd((unsigned long long*)&ctl->live_groups, (u64)s_ins);
  if (LEAF && d.split && threadIdx.x == 0) {
    // the last CTA to finish leaves the batch's errors so far for the split
    // placement (the block barrier above orders this CTA's raises before the
    // fence; the other CTAs fenced theirs before counting)
    __threadfence();
    if (atomicAdd(&ctl->fin_ctr, 1u) == gridDim.x - 1) {
      __threadfence();
      ctl->fin_ctr = 0;
      ctl->pre_err = *(volatile int*)&ctl->batch_err;
      ctl->n_done_leaf = *(volatile u32*)&ctl->n_done;  // the upper levels append after these
    }
  }
}

// ---------------------------------------------------------------------------
// Streaming release with the CONCAT level M above the leaf parent (Sec. 3.2).
// A group of level M receives its children as spans: a level-(M+1) group
// that completes appends its concatenation to its parent's buffer.  Right
// after level M has run, so that its touched list is still there:
//   k_up_meta      the spans handed up in this batch get their meta entry
//                  {child index, payload position} in the parent's buffer,
//                  whose room the parent's finalize allocated;
//   k_up_release   a warp per touched group of level M left open marks its
//                  buffered children from `rel` on and finds the first one
//                  missing: a run that grew is a partial release (a done
//                  entry of its own, buffered children released);
//   k_up_rel_seq   a release's completion seq is the latest among its
//                  children completed in this batch (the one at `rel` is
//                  one of them, or the run could not have grown);
//   k_up_rel_mask  the releases take their places in the emission order.
// The records scan, placement, gather, records and buffer compaction then
// treat a release as at the leaf parent.
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(kThreads) k_up_meta(Dev d) {
  pdl_enter();
  Ctl* ctl = d.ctl;
  if (poisoned(ctl)) return;
  if (*(const volatile int*)&ctl->batch_err) return;  // a parent entry may be unusable
  const int M = d.cfg.concat_level;
  const u32 nd = min(ctl->n_done, d.sc.done_cap);
  for (u32 di = gtid(); di < nd; di += gstride()) {
    if ((int)d.sc.done_lvl[di] != M + 1) continue;
    const u32 e = d.sc.done_e[di] & d.tab.mask;
    const u32 P = d.tab.par[e] & d.tab.mask;
    const u64 ap = d.tab.app[e];
    const u64 m = ap >> 40;
    if (m >= d.tab.vec_n[2 * (u64)P]) continue;
    bool ok;
    const u64 a = vec_addr(d.tab, P, 0, 2 * m, &ok);
    if (!ok) continue;
    d.ar.pool[a] = (int32_t)d.tab.cidx[e];
    d.ar.pool[a + 1] = (int32_t)(u32)(ap & kPos40);
  }
}

// `list`: level M's touched entries; with `seg_start`, the entries are the
// sorted keys at the segment starts instead (a TOPK level M).
__global__ void __launch_bounds__(kThreads) k_up_release(Dev d, const u32* list, const u32* seg_start) {
  pdl_enter();
  Ctl* ctl = d.ctl;
  if (poisoned(ctl)) return;
  if (*(const volatile int*)&ctl->batch_err) return;
  const int M = d.cfg.concat_level;
  const u32 nt = min(ctl->n_segs[M], d.cfg.n_max);
  const u32 ep = ctl->epoch;
  const int lane = threadIdx.x & 31;
  const u32 gw = gtid() >> 5, nw = gstride() >> 5;
  for (u32 w = gw; w < nt; w += nw) {
    const u32 e = (seg_start ? list[seg_start[w]] : list[w]) & d.tab.mask;
    if (d.tab.hot[e].done_epoch == ep) continue;  // completed by this batch: its final record
    const u32 rel = d.tab.rel[e];
    const u32 B = d.tab.vec_n[2 * (u64)e];
    if (B == 0) continue;
    // B buffered children cannot fill B + 1 bits: the run ends inside the map
    const u64 words = (u64)B / 32 + 1;
    unsigned long long base = 0;
    if (lane == 0) base = atomicAdd((unsigned long long*)&ctl->bm_used, (unsigned long long)words);
    base = __shfl_sync(0xFFFFFFFFu, base, 0);
    if (base + words > d.sc.bm_cap) {
      if (lane == 0) raise_err(ctl, ALTO_ENOSPC);
      continue;
    }
    u32* bm = d.sc.bm + base;
    for (u64 x = lane; x < words; x += 32) bm[x] = 0;
    __syncwarp();
    const u64 span = words * 32;
    for (u32 k = lane; k < B; k += 32) {
      bool ok;
      const u64 a = vec_addr(d.tab, e, 0, 2 * (u64)k, &ok);
      if (!ok) continue;
      const u32 c = (u32)d.ar.pool[a];
      if (c >= rel && (u64)(c - rel) < span) atomicOr(&bm[(c - rel) >> 5], 1u << ((c - rel) & 31));
    }
    __syncwarp();
    u32 z = kNone;
    for (u64 wb = 0; wb < words && z == kNone; wb += 32) {
      const u64 x = wb + lane;
      u32 cand = kNone;
      if (x < words) {
        const u32 free_bits = ~__ldcg(&bm[x]);
        if (free_bits) cand = (u32)(x * 32) + (u32)(__ffs(free_bits) - 1);
      }
      z = __reduce_min_sync(0xFFFFFFFFu, cand);
    }
    if (z == kNone || z == 0) continue;  // child `rel` is still missing (or no room)
    if (lane == 0) {
      const u32 di = atomicAdd(&ctl->n_done, 1u);
      const u32 q = atomicAdd(&ctl->n_rel, 1u);
      if (di < d.sc.done_cap && q < d.cfg.n_max) {
        d.sc.done_e[di] = e;
        d.sc.done_lvl[di] = (u32)M;
        d.sc.done_cseq[di] = 0;
        d.sc.done_part[di] = 2u;  // every released child was buffered: the buffer is compacted
        d.tab.rnew[e] = rel + z;
        d.tab.hot[e].done_epoch = ep;
        d.tab.done_idx[e] = di;
        d.sc.rel_seg[q] = di;
      } else {
        raise_err(ctl, ALTO_ENOSPC);
      }
    }
  }
}

__global__ void __launch_bounds__(kThreads) k_up_rel_seq(Dev d) {
  pdl_enter();
  Ctl* ctl = d.ctl;
  if (poisoned(ctl) || *(const volatile int*)&ctl->batch_err) return;
  const int M = d.cfg.concat_level;
  const u32 ep = ctl->epoch;
  const u32 nd = min(ctl->n_done, d.sc.done_cap);
  for (u32 di = gtid(); di < nd; di += gstride()) {
    if ((int)d.sc.done_lvl[di] != M + 1) continue;
    const u32 e = d.sc.done_e[di] & d.tab.mask;
    const u32 P = d.tab.par[e] & d.tab.mask;
    if (d.tab.hot[P].done_epoch != ep) continue;
    const u32 dp = d.tab.done_idx[P];
    if (dp >= nd || d.sc.done_part[dp] != 2u) continue;
    const u32 c = d.tab.cidx[e];
    if (c >= d.tab.rel[P] && c < d.tab.rnew[P]) atomicMax(&d.sc.done_cseq[dp], d.sc.done_cseq[di]);
  }
}

__global__ void __launch_bounds__(kThreads) k_up_rel_mask(Dev d) {
  pdl_enter();
  Ctl* ctl = d.ctl;
  if (poisoned(ctl) || *(const volatile int*)&ctl->batch_err) return;
  const int D = d.cfg.depth, M = d.cfg.concat_level;
  const u32 nr = min(ctl->n_rel, d.cfg.n_max);
  const u32 nd = min(ctl->n_done, d.sc.done_cap);
  for (u32 q = gtid(); q < nr; q += gstride()) {
    const u32 di = d.sc.rel_seg[q];
    if (di >= nd) continue;
    const u32 cs = d.sc.done_cseq[di];
    if (cs < ctl->n) {
      atomicOr(&d.sc.mask[cs], 1u << (D - 1 - M));
      atomicAdd(&d.sc.mblk[cs >> 5], 1u);
    }
  }
}

// Emission rank of each completed group: records completed at earlier
// arrival indices, plus the deeper groups completed at the same index.  The
// scan runs over runs of 32 seqs (their completion counts); a group adds the
// completions of its run's earlier seqs from the per-seq level masks.
struct RankScan {
  const u32* mblk;
  u32* prefix;
  const u32* n_dev;
  __device__ u64 size(const Ctl*) const { return (*n_dev + 31) >> 5; }
  __device__ u64 value(u64 i) const { return mblk[i]; }
  // only runs that completed a group are ever looked up
  __device__ void out(u64 i, u64 excl, u64 v) const {
    if (v) prefix[i] = (u32)excl;
  }
  __device__ void total(Ctl* ctl, u64 t) const { ctl->n_emit = t; }
};

__global__ void __launch_bounds__(kThreads) k_done_rank(Dev d) {
  pdl_enter();
  Ctl* ctl = d.ctl;
  if (poisoned(ctl)) return;
  const int D = d.cfg.depth, M = d.cfg.concat_level;
  const u32 nd = min(ctl->n_done, d.sc.done_cap);
  for (u32 di = gtid(); di < nd; di += gstride()) {
    const u32 e = d.sc.done_e[di];
    const int l = (int)d.sc.done_lvl[di];
    const u32 cs = d.sc.done_cseq[di];
    const int bit = D - 1 - l;
    u32 r = kNone;
    if (cs < ctl->n) {
      // the run's earlier seqs: its 32 masks are one 128-byte line
      const u32 b0 = cs & ~31u;
      const uint4* m4 = reinterpret_cast<const uint4*>(d.sc.mask + b0);
      u32 before = 0;
#pragma unroll
      for (int q = 0; q < 8; ++q) {
        const uint4 v = m4[q];
        const u32 s0 = b0 + 4 * q;
        before += (s0 < cs ? __popc(v.x) : 0) + (s0 + 1 < cs ? __popc(v.y) : 0) +
                  (s0 + 2 < cs ? __popc(v.z) : 0) + (s0 + 3 < cs ? __popc(v.w) : 0);
      }
      r = d.sc.prefix[cs >> 5] + before + __popc(d.sc.mask[cs] & ((1u << bit) - 1u));
    }
    if (r >= nd) {
      raise_err(ctl, ALTO_EINCONSIST);
      d.sc.done_rank[di] = kNone;
      continue;
    }
    d.sc.done_rank[di] = r;
    d.sc.r_done[r] = di;
    const u32 nch = d.tab.hot[e].last + 1;
    // streaming: children rel.. of the run that ends this batch (all of them
    // up to the last for a final record); a partial record has no top-k
    const bool part = d.cfg.stream && d.sc.done_part[di];
    const u32 rel = (d.cfg.stream && l == M) ? d.tab.rel[e] : 0u;
    const u32 rend = part ? d.tab.rnew[e] : nch;
    d.sc.r_dense_n[r] = (l == M) ? rend - rel : 0u;
    d.sc.r_topk_n[r] = (!part && d.cfg.score_op[l] == ALTO_SCORE_TOPK) ? min(nch, (u32)d.cfg.topk_k[l]) : 0u;
    d.sc.r_meta_n[r] = (l == M) ? d.tab.vec_n[2 * (u64)e] : 0u;
    // a leaf parent of the CONCAT level: where this batch's leaves go is its
    // dense base, r_dense_base[r] once the record scans ran (mode 4: by rank;
    // the scans then write no per-entry state)
    if (l == M && M == D - 1 && !d.split) d.tab.bstate[e] = make_uint4(ctl->epoch, 4u, r, 0u);
  }
}

// Exclusive scan of a per-record u32 count into u64 offsets.
struct CountScan {
  const u32* in;
  u64* out_off;
  const u32* n_dev;
  u32 cap;
  int which;  // 0 dense, 1 topk, 2 arena; split placement: 3 unused, 4 dense, 5 arena
  // dense only: also leave each completing group's first slot in its entry
  const u32* r_done = nullptr;
  const u32* done_e = nullptr;
  u64* dbase = nullptr;
  u32 tmask = 0;
  uint4* bstate = nullptr;
  const Ctl* ctlp = nullptr;
  __device__ u64 size(const Ctl*) const { return min(*n_dev, cap); }
  __device__ u64 value(u64 i) const { return in[i]; }
  __device__ void out(u64 i, u64 excl, u64 v) const {
    out_off[i] = excl;
    if (dbase && v) {
      const u32 di = r_done[i];
      if (di < cap) {
        const u32 e = done_e[di] & tmask;
        dbase[e] = excl;
        if (bstate && !ctlp->skip_dense)
          bstate[e] = make_uint4(ctlp->epoch, 2u, (u32)excl, (u32)(excl >> 32));
      }
    }
  }
  __device__ void total(Ctl* ctl, u64 t) const {
    if (which == 3) return;  // an unused scan of a three-scan launch
    out_off[size(nullptr)] = t;
    if (which == 0) ctl->dense_total = t;
    else if (which == 1) ctl->topk_total = t;
    else if (which == 2) ctl->arena_total = t;
    else if (which == 4) ctl->leaf_dense_total = t;
    else ctl->leaf_arena_total = t;
  }
};

// Levels M < l: dense slots (which 0) and buffered spans (which 1) of the
// groups completing in this batch, over the done list; which 2 is empty.
// Their dense region follows level M's.  The slot scan also leaves each such
// group's first slot in its entry (and, for a leaf parent, where this batch's
// leaves go) and writes the group's meta entry {child index, payload
// position} into its parent's vectors, whose chunks the parent's finalize
// allocated.
struct ChainScan {
  const u32* done_e;
  const u32* done_lvl;
  const u32* n_dev;
  u32 cap;
  int which;
  u64* out_off;
  Table tab;
  int32_t* arena_pool;
  Ctl* ctlp;
  int M, L;
  __device__ u64 size(const Ctl*) const { return (which == 2) ? 0 : min(*n_dev, cap); }
  __device__ u64 value(u64 i) const {
    if ((int)done_lvl[i] <= M) return 0;
    const u32 e = done_e[i] & tab.mask;
    return (which == 0) ? (u64)tab.hot[e].last + 1 : (u64)tab.vec_n[2 * (u64)e];
  }
  __device__ void out(u64 i, u64 excl, u64 v) const {
    if (which == 2) return;
    const u64 off = (which == 0) ? ctlp->dense_total : 0;
    out_off[i] = off + excl;
    if (which != 0 || v == 0) return;
    const u32 e = done_e[i] & tab.mask;
    const u64 base = off + excl;
    tab.dbase[e] = base;
    if ((int)done_lvl[i] == L)
      tab.bstate[e] = make_uint4(ctlp->epoch, 2u, (u32)base, (u32)(base >> 32));
    if (*(const volatile int*)&ctlp->batch_err) return;  // a parent entry may be unusable
    const u32 P = tab.par[e] & tab.mask;
    const u64 ap = tab.app[e];
    const u64 m = ap >> 40;
    if (m >= tab.vec_n[2 * (u64)P]) return;
    bool ok;
    const u64 a = vec_addr(tab, P, 0, 2 * m, &ok);
    if (!ok) return;
    arena_pool[a] = (int32_t)tab.cidx[e];
    arena_pool[a + 1] = (int32_t)(u32)(ap & kPos40);
  }
  __device__ void total(Ctl* ctl, u64 t) const {
    if (which == 2) return;
    const u64 off = (which == 0) ? ctl->dense_total : 0;
    out_off[size(ctl)] = off + t;
    if (which == 0) ctl->chain_total = t;
    else ctl->chain_arena = t;
  }
};

// The batch's output sizes against the capacities, once the record scans
// have their totals; run by the last CTA of the record-offset scans (volatile
// reads: other CTAs wrote the totals).
struct CapCheck {
  static constexpr bool kActive = true;
  static constexpr bool kSide = false;
  u64 out_records, dense_cap, out_topk, done_cap;
  // split placement: the placement beside these scans checks the dense slots
  // and the payload itself, and only the records stand down here
  bool split = false;
  __device__ void operator()(Ctl* ctl) const {
    volatile Ctl* v = ctl;
    if (v->status != ALTO_OK || v->abort) return;
    bool bad = false;
    if (v->rec_count + v->n_done > out_records) bad = true;
    if (v->dense_total + v->chain_total > dense_cap) bad = true;
    if (v->topk_count + v->topk_total > out_topk) bad = true;
    if (v->n_done > done_cap) bad = true;
    if (bad) {
      raise_err(ctl, ALTO_ENOSPC);
      v->skip_rec = 1;
      if (!split) v->skip_dense = 1;
    }
    // allocations of the level kernels may have taken a free stack below zero
    for (int j = 0; j < kNumChunks; ++j)
      if (v->top[j] < 0) v->top[j] = 0;
  }
};

// Split placement, first step: the leaf parents completing before each run
// of 32 arrival indices (the leaf finalize counted them per run).
struct LeafRunScan {
  const u32* lblk;
  u32* lprefix;
  __device__ u64 size(const Ctl* ctl) const { return (ctl->n + 31) >> 5; }
  __device__ u64 value(u64 i) const { return lblk[i]; }
  // only runs that completed a leaf parent are ever looked up
  __device__ void out(u64 i, u64 excl, u64 v) const {
    if (v) lprefix[i] = (u32)excl;
  }
  __device__ void total(Ctl*, u64) const {}
};

// Split placement: each leaf parent's rank among the leaf parents completing
// in the batch (their emission order restricted to the leaf level: by
// completion seq, at most one a seq), its children and buffered spans by
// that rank, and its placement state (mode 4: its dense base by rank).  The
// leaf parents are the done list's first n_done_leaf entries; the upper
// levels append theirs, and set other bits of the masks, beside this kernel.
__global__ void __launch_bounds__(kThreads) k_leaf_rank(Dev d) {
  pdl_enter();
  Ctl* ctl = d.ctl;
  if (halted(ctl)) return;
  const u32 nl = min(ctl->n_done_leaf, d.sc.done_cap);
  for (u32 di = gtid(); di < nl; di += gstride()) {
    const u32 e = d.sc.done_e[di] & d.tab.mask;
    const u32 cs = d.sc.done_cseq[di];
    if (cs >= ctl->n) continue;
    const u32 b0 = cs & ~31u;
    const uint4* m4 = reinterpret_cast<const uint4*>(d.sc.mask + b0);
    u32 before = 0;
#pragma unroll
    for (int q = 0; q < 8; ++q) {
      const uint4 v = m4[q];
      const u32 s0 = b0 + 4 * q;
      before += (s0 < cs ? (v.x & 1u) : 0) + (s0 + 1 < cs ? (v.y & 1u) : 0) + (s0 + 2 < cs ? (v.z & 1u) : 0) +
                (s0 + 3 < cs ? (v.w & 1u) : 0);
    }
    const u32 r = d.sc.lprefix[cs >> 5] + before;
    // the run's count is consumed (the next batch starts from zero)
    d.sc.lblk[cs >> 5] = 0;
    if (r >= nl) continue;
    d.sc.l_done[r] = di;
    d.sc.l_dense_n[r] = d.tab.hot[e].last + 1;
    d.sc.l_meta_n[r] = d.tab.vec_n[2 * (u64)e];
    d.tab.bstate[e] = make_uint4(ctl->epoch, 4u, r, 0u);
  }
}

// The split placement's dense slots against their capacity, once its scans
// have their totals (the placement, the length scan and the gather then
// stand down).
struct LeafCheck {
  static constexpr bool kActive = true;
  static constexpr bool kSide = true;
  u64 dense_cap;
  __device__ void operator()(Ctl* ctl) const {
    volatile Ctl* v = ctl;
    if (v->status != ALTO_OK || v->abort) return;
    if (v->leaf_dense_total > dense_cap) {
      raise_err(ctl, ALTO_ENOSPC);
      v->skip_dense = 1;
    }
  }
};

// Payload lengths of the leaves in sorted order, scanned: a leaf's position
// inside its group's new arena data.
struct LenScan {
  const u32* perm;
  const u32* off;
  u64* out_scan;
  const u32* n_dev;
  __device__ u64 size(const Ctl*) const { return *n_dev; }
  __device__ u64 value(u64 j) const {
    u32 i = perm[j];
    return off[i + 1] - off[i];
  }
  __device__ void out(u64 j, u64 excl, u64) const { out_scan[j] = excl; }
  __device__ void total(Ctl*, u64 t) const { out_scan[size(nullptr)] = t; }
};

// TOPK leaf level: chunks for the arena ranges reserved by this batch's open
// CONCAT groups (the reduce recorded their old sizes per segment).  A block
// counts its requests per size class in shared memory and takes them from the
// class's free stack (or the bump allocator) with one atomic each.  (Without
// TOPK the leaf finalize allocates these itself, per warp.)
constexpr int kMaxReq = 8;

__global__ void __launch_bounds__(kThreads) k_carry_alloc(Dev d) {
  pdl_enter();
  Ctl* ctl = d.ctl;
  if (no_copy(ctl)) return;
  __shared__ u32 s_cnt[kNumChunks];
  __shared__ int s_old[kNumChunks];
  __shared__ u32 s_avail[kNumChunks];
  __shared__ u64 s_bump[kNumChunks];
  __shared__ unsigned long long s_used;
  const u32 nseg = min(ctl->n_segs[d.cfg.depth - 1], d.cfg.n_max);
  for (u32 base = blockIdx.x * blockDim.x; base < nseg; base += gridDim.x * blockDim.x) {
    if (threadIdx.x < kNumChunks) s_cnt[threadIdx.x] = 0;
    if (threadIdx.x == 0) s_used = 0;
    __syncthreads();
    const u32 s = base + threadIdx.x;
    u32 e = 0;
    int nreq = 0;
    uint8_t rvec[kMaxReq], rj[kMaxReq];
    u32 rr[kMaxReq];
    bool want = false;
    u64 old0 = 0, old1 = 0;
    if (s < nseg && (d.sc.seg_carry[s] == 1u || d.sc.seg_carry[s] == 3u)) {
      e = d.sc.leaf_keys[d.sc.leaf_seg_start[s]] & d.tab.mask;
      want = true;
      old0 = d.sc.seg_vb0[s];
      old1 = d.sc.seg_vb1[s];
    }
    if (want) {
      for (int vec = 0; vec < kVecs; ++vec) {
        const u64 mult = (vec == 0) ? 2 : 1;
        const u64 old_el = ((vec == 0) ? old0 : old1) * mult;
        const u64 new_el = (u64)d.tab.vec_n[2 * (u64)e + vec] * mult;
        if (new_el <= old_el) continue;
        const int jf = (old_el == 0) ? 0 : chunk_of(old_el - 1) + 1;
        const int jl = chunk_of(new_el - 1);
        if (jl >= kNumChunks) raise_err(ctl, ALTO_ENOSPC);
        for (int j = jf; j <= jl && j < kNumChunks; ++j) {
          if (nreq < kMaxReq) {
            rvec[nreq] = (uint8_t)vec;
            rj[nreq] = (uint8_t)j;
            rr[nreq] = atomicAdd(&s_cnt[j], 1u);
            ++nreq;
          } else {  // rare: a vector grew by many classes at once
            u32 c = alloc_chunk(d.ar, ctl, j);
            d.tab.dir[((u64)e * kVecs + vec) * kNumChunks + j] = c;
            if (c != kNone) atomicAdd(&s_used, (unsigned long long)chunk_size(j));
          }
        }
      }
    }
    __syncthreads();
    if (threadIdx.x < kNumChunks) {
      const int j = threadIdx.x;
      const u32 cnt = s_cnt[j];
      if (cnt) {
        const int old = atomicSub(&ctl->top[j], (int)cnt);
        const u32 avail = (old <= 0) ? 0u : min((u32)old, cnt);
        s_old[j] = old;
        s_avail[j] = avail;
        if (cnt > avail)
          s_bump[j] = atomicAdd((unsigned long long*)&ctl->bump,
                                (unsigned long long)((cnt - avail) * chunk_size(j)));
      }
    }
    __syncthreads();
    for (int q = 0; q < nreq; ++q) {
      const int j = rj[q];
      const u32 r = rr[q];
      u32 c;
      if (r < s_avail[j]) {
        c = d.ar.stack[d.ar.stack_off[j] + (u64)(s_old[j] - 1 - (int)r)];
      } else {
        const u64 o = s_bump[j] + (u64)(r - s_avail[j]) * chunk_size(j);
        if (o + chunk_size(j) > d.ar.elems) {
          raise_err(ctl, ALTO_ENOSPC);
          c = kNone;
        } else {
          c = (u32)o;
        }
      }
      d.tab.dir[((u64)e * kVecs + rvec[q]) * kNumChunks + j] = c;
      if (c != kNone) atomicAdd(&s_used, (unsigned long long)chunk_size(j));
    }
    __syncthreads();
    if (threadIdx.x == 0 && s_used) atomicAdd((unsigned long long*)&ctl->arena_used, s_used);
  }
}

__global__ void k_fix_tops(Ctl* ctl) {
  pdl_enter();
  int j = threadIdx.x;
  if (j < kNumChunks && ctl->top[j] < 0) ctl->top[j] = 0;
}

// Append the leaves of open CONCAT groups to their arena vectors: eight lanes
// per leaf, over the sorted leaves.  A leaf's vector position is its group's
// reserved base plus its offset inside the segment (written by the reduce;
// for a partial release, among the leaves it keeps).  (A lane per leaf with
// the spans then copied four at a time, as in the gather, measured slower;
// so did a warp per carried segment, which leaves a hot group's tens of
// thousands of leaves to one warp.)
template <bool G>
__global__ void __launch_bounds__(kThreads) k_carry_copy(Dev d, Batch bv) {
  pdl_enter();
  const Batch b = batch_of<G>(bv, d);
  Ctl* ctl = d.ctl;
  if (no_copy(ctl)) return;
  const int D = d.cfg.depth;
  const u64 n = b.n;
  const u32 nseg = min(ctl->n_segs[D - 1], d.cfg.n_max);
  const u32 sub = threadIdx.x & 7;
  const u32 g0 = gtid() >> 3, ng = gstride() >> 3;
  for (u32 j = g0; j < b.n; j += ng) {
    const u32 s = d.sc.leaf_seg_of[j];
    if (s >= nseg) continue;
    const u32 sc_mode = d.sc.seg_carry[s];
    if (sc_mode != 1u && sc_mode != 3u) continue;
    const u32 i = d.sc.leaf_perm[j];
    if (i >= b.n) continue;
    const u32 e = d.sc.leaf_keys[j] & d.tab.mask;
    const u32 s0 = d.sc.leaf_seg_start[s];
    if (s0 > j) continue;
    // a partial release buffers only the leaves it keeps
    const u32 mr = (sc_mode == 3u) ? d.sc.leaf_mrank[j] : j - s0;
    if (mr == kNone) continue;
    const u32 o0 = b.off[i];
    const u32 len = b.off[i + 1] - o0;
    const u64 mpos = (u64)d.sc.seg_vb0[s] + mr;
    const u64 ppos = (u64)d.sc.seg_vb1[s] + d.sc.leaf_pos[j];
    if (mpos >= d.tab.vec_n[2 * (u64)e] || ppos + len > d.tab.vec_n[2 * (u64)e + 1] ||
        (u64)o0 + len > b.n_payload)
      continue;
    bool ok;
    if (sub == 0) {
      const u64 a = vec_addr(d.tab, e, 0, 2 * mpos, &ok);
      if (ok) {
        d.ar.pool[a] = (int32_t)tag_child(b.tags[(u64)(D - 1) * n + i]);
        d.ar.pool[a + 1] = (int32_t)(u32)ppos;
      }
    }
    for (u32 k = sub; k < len; k += 8) {
      const u64 a = vec_addr(d.tab, e, 1, ppos + k, &ok);
      if (ok) d.ar.pool[a] = b.pay[o0 + k];
    }
  }
}

// Dense child slots of completing CONCAT groups, from this batch's leaves
// (and, streaming, of the leaves a partial release takes from the batch).
template <bool G>
__global__ void __launch_bounds__(kThreads) k_dense_batch(Dev d, Batch bv) {
  pdl_enter();
  const Batch b = batch_of<G>(bv, d);
  Ctl* ctl = d.ctl;
  if (no_copy(ctl) || ctl->skip_dense) return;
  const int D = d.cfg.depth, M = d.cfg.concat_level;
  const u32 ep = ctl->epoch;
  const u64 n = b.n;
  const u32 nd = min(ctl->n_done, d.sc.done_cap);
  const u32 nseg = min(ctl->n_segs[D - 1], d.cfg.n_max);
  for (u32 j = gtid(); j < b.n; j += gstride()) {
    const u32 s = d.sc.leaf_seg_of[j];
    if (s >= nseg) continue;
    const u32 sc_mode = d.sc.seg_carry[s];
    if (sc_mode != 2u && sc_mode != 3u) continue;
    const u32 e = d.sc.leaf_keys[j] & d.tab.mask;
    const u32 i = d.sc.leaf_perm[j];
    if (i >= b.n || d.tab.hot[e].done_epoch != ep) continue;
    const u32 di = d.tab.done_idx[e];
    if (di >= nd) continue;
    const u32 c = tag_child(b.tags[(u64)(D - 1) * n + i]);
    if (c > d.tab.hot[e].last) continue;
    const u32 rel = d.cfg.stream_leaf ? d.tab.rel[e] : 0u;  // children below were released earlier
    if (c < rel) continue;
    if (sc_mode == 3u && c >= d.tab.rnew[e]) continue;   // kept in the buffer
    // the group's first slot: by rank at the CONCAT level, from the chain
    // scan below it
    const u32 rk = d.sc.done_rank[di];
    if (M == D - 1 && rk >= nd) continue;
    const u64 slot = ((M == D - 1) ? d.sc.r_dense_base[rk] : d.tab.dbase[e]) + (c - rel);
    if (slot >= d.cfg.dense_cap) continue;
    const u32 old = atomicExch(&d.sc.dense[slot].x, ep);
    if (old == ep) raise_err(ctl, ALTO_EDUP);
    const u32 o0 = b.off[i];
    d.sc.dense[slot].y = b.off[i + 1] - o0;
    d.sc.dense[slot].z = kNone;
    d.sc.dense[slot].w = o0;
  }
}

// Dense child slots from the arena: spans buffered by earlier batches (and,
// above the leaf parent, handed up earlier in this batch).  LEVEL_M: the
// groups of level M, by emission rank; otherwise the groups of levels M < l,
// by done index.  (A warp per group with buffered spans, in place of the
// binary search, measured slower: a few groups hold most of the spans.)
template <bool LEVEL_M, bool SPLIT = false>
__device__ __forceinline__ void dense_arena_body(const Dev& d, Ctl* ctl, u64 first, u64 stride) {
  const u32 ep = ctl->epoch;
  // split placement: the leaf parents by their rank among themselves (the
  // done list grows beside it)
  const u32 nd = min(SPLIT ? ctl->n_done_leaf : ctl->n_done, d.sc.done_cap);
  const u64 na = SPLIT ? ctl->leaf_arena_total : LEVEL_M ? ctl->arena_total : ctl->chain_arena;
  const u64* abase = SPLIT ? d.sc.l_arena_base : LEVEL_M ? d.sc.r_arena_base : d.sc.c_arena_base;
  const u32* by_rank = SPLIT ? d.sc.l_done : d.sc.r_done;
  const u32* meta_n = SPLIT ? d.sc.l_meta_n : d.sc.r_meta_n;
  const u64* dense_base = SPLIT ? d.sc.l_dense_base : d.sc.r_dense_base;
  for (u64 a = first; a < na; a += stride) {
    // last index x with abase[x] <= a: the one whose spans contain a
    u32 lo = 0, hi = nd;
    while (hi - lo > 1) {
      u32 mid = (lo + hi) >> 1;
      if (abase[mid] <= a) lo = mid;
      else hi = mid;
    }
    const u32 di = LEVEL_M ? by_rank[lo] : lo;
    if (di >= nd) continue;
    if (!LEVEL_M && (int)d.sc.done_lvl[di] <= d.cfg.concat_level) continue;
    const u32 e = d.sc.done_e[di] & d.tab.mask;
    const u64 k = a - abase[lo];
    const u32 mn = LEVEL_M ? meta_n[lo] : d.tab.vec_n[2 * (u64)e];
    const u64 dbase = LEVEL_M ? dense_base[lo] : d.tab.dbase[e];
    if (k >= mn) continue;
    bool ok1, ok2 = true;
    u64 ma = vec_addr(d.tab, e, 0, 2 * k, &ok1);
    if (!ok1) continue;
    const u32 c = (u32)d.ar.pool[ma];
    const u32 pos = (u32)d.ar.pool[ma + 1];
    u32 end;
    if (k + 1 < mn) {
      u64 na2 = vec_addr(d.tab, e, 0, 2 * (k + 1) + 1, &ok2);
      end = ok2 ? (u32)d.ar.pool[na2] : pos;
    } else {
      end = d.tab.vec_n[2 * (u64)e + 1];
    }
    // streaming: the buffer holds children rel.. only; a partial release
    // places those below rnew and keeps the rest
    const u32 rel = (LEVEL_M && d.cfg.stream) ? d.tab.rel[e] : 0u;
    if (c > d.tab.hot[e].last || end < pos || c < rel) {
      raise_err(ctl, ALTO_EDUP);
      continue;
    }
    if (LEVEL_M && d.cfg.stream && d.sc.done_part[di] && c >= d.tab.rnew[e]) continue;
    // level M: its first dense slot by rank (split: by its rank among the
    // leaf parents); the levels below: by done index
    const u64 slot = dbase + (c - rel);
    if (slot >= d.cfg.dense_cap) continue;
    u32 old = atomicExch(&d.sc.dense[slot].x, ep);
    if (old == ep) raise_err(ctl, ALTO_EDUP);
    d.sc.dense[slot].y = end - pos;
    d.sc.dense[slot].z = e;
    d.sc.dense[slot].w = pos;
  }
}

// Leaf level without TOPK, per fragment in arrival order, eight lanes each:
// a fragment of a group left open takes its arena position from the group's
// cursor (one 64-bit atomic: leaf index and payload offset together) and is
// copied there; a fragment of a group completed by this batch is placed at
// its dense child slot.
// PART 1: only the fragments of groups left open (their arena copies need
// nothing after the leaf finalize, so they may run beside the upper levels);
// PART 2: only the dense slots (this batch's fragments and the buffered
// children of the completing groups); PART 3: both.
template <bool G, int PART>
__global__ void __launch_bounds__(kThreads, 8) k_leaf_place(Dev d, Batch bv) {
  pdl_enter();
  const Batch b = batch_of<G>(bv, d);
  Ctl* ctl = d.ctl;
  if (stand_down(d, ctl)) return;
  const int D = d.cfg.depth;
  const u32 ep = ctl->epoch;
  const u64 n = b.n;
  const bool dense_ok = !ctl->skip_dense;
  const u64 dcap = d.cfg.dense_cap;
  const int lane = threadIdx.x & 31;
  const u32 end = (b.n + 31) & ~31u;  // whole warps iterate together
  for (u32 i = gtid(); i < end; i += gstride()) {
    u32 e = 0, mode = 0;  // 1 arena, 2 dense
    u32 o0 = 0, len = 0, c = 0;
    uint4 bs = make_uint4(0, 0, 0, 0);
    if (i < b.n) {
      // the fragment's own fields do not depend on its group: load them first
      e = d.sc.leaf_sort_keys0[i] & d.tab.mask;
      o0 = b.off[i];
      len = b.off[i + 1] - o0;
      c = tag_child(b.tags[(u64)(D - 1) * n + i]);
      bs = d.tab.bstate[e];
      if (bs.x == ep) mode = bs.y;
      u64 base = ((u64)bs.w << 32) | bs.z;
      if (mode == 4) {
        // a CONCAT-level leaf parent stamped with its rank: its dense base
        // (the carried-leaves-only launch may run before the record scans,
        // and does not need it)
        mode = 2;
        if (PART & 2) base = (bs.z < d.sc.done_cap) ? (d.split ? d.sc.l_dense_base : d.sc.r_dense_base)[bs.z] : dcap;
      }
      bs.z = (u32)base;
      bs.w = (u32)(base >> 32);
      if (mode == 2 && !dense_ok) mode = 0;
      if (!(PART & mode)) mode = 0;  // mode 1 is PART bit 1, mode 2 PART bit 2
    }
    if (mode == 2) {
      // every child index is below n_children (checked at completion); a
      // repeated child leaves some other slot unfilled, which the length
      // scan reports
      const u64 slot = (((u64)bs.w << 32) | bs.z) + c;
      if (slot < dcap) d.sc.dense[slot] = make_uint4(ep, len, kNone, o0);
    }
    u64 ppos = 0;
    bool copy = false;
    if (mode == 1) {
      const u64 old = atomicAdd((unsigned long long*)&d.tab.cur[e], (1ull << 40) | len);
      const u64 mpos = old >> 40;
      ppos = old & ((1ull << 40) - 1);
      if (mpos < d.tab.vec_n[2 * (u64)e] && ppos + len <= d.tab.vec_n[2 * (u64)e + 1] &&
          (u64)o0 + len <= b.n_payload) {
        bool ok;
        const u64 a = vec_addr(d.tab, e, 0, 2 * mpos, &ok);
        if (ok) {
          d.ar.pool[a] = (int32_t)c;
          d.ar.pool[a + 1] = (int32_t)(u32)ppos;
        }
        copy = true;
      }
    }
    // arena-bound fragments: eight lanes copy one span, four spans at a time,
    // the first 64 elements' loads all issued before the stores (as in the
    // gather); the span's first chunk is looked up once, elements past it
    // one by one
    u32 pending = __ballot_sync(0xFFFFFFFFu, copy);
    const int sub = lane & 7, grp = lane >> 3;
    while (pending) {
      u32 pm = pending;  // this group's span: the grp-th pending lane
      for (int k = 0; k < grp; ++k) pm &= pm - 1;
      for (int k = 0; k < 4; ++k) pending &= pending - 1;
      const int src = pm ? __ffs(pm) - 1 : 0;
      const u32 se = __shfl_sync(0xFFFFFFFFu, e, src);
      const u32 so = __shfl_sync(0xFFFFFFFFu, o0, src);
      const u32 sl0 = __shfl_sync(0xFFFFFFFFu, len, src);
      const u64 sp = __shfl_sync(0xFFFFFFFFu, ppos, src);
      const u32 sl = pm ? sl0 : 0u;
      if (sl == 0) continue;
      const int j1 = chunk_of(sp);
      const u64 room = chunk_start(j1) + chunk_size(j1) - sp;
      bool ok1;
      const u64 a1 = vec_addr(d.tab, se, 1, sp, &ok1);
      const u32 n1 = ok1 ? ((room < sl) ? (u32)room : sl) : 0u;
      const int32_t* src_p = b.pay + so;
      int32_t* dst_p = d.ar.pool + a1;
      int32_t v[8];
#pragma unroll
      for (int q = 0; q < 8; ++q) {
        const u32 k = sub + 8 * q;
        v[q] = (k < n1) ? src_p[k] : 0;
      }
#pragma unroll
      for (int q = 0; q < 8; ++q) {
        const u32 k = sub + 8 * q;
        if (k < n1) dst_p[k] = v[q];
      }
      for (u32 k = 64 + sub; k < n1; k += 8) dst_p[k] = src_p[k];
      for (u32 k = n1 + sub; k < sl; k += 8) {
        bool ok;
        const u64 a = vec_addr(d.tab, se, 1, sp + k, &ok);
        if (ok) d.ar.pool[a] = src_p[k];
      }
    }
  }
  // the completing groups' children buffered by earlier batches take their
  // dense slots in the same launch: other slots than the fragments' above,
  // and their latency overlaps that of the fragments
  if ((PART & 2) && !ctl->skip_dense) {
    if (d.split) dense_arena_body<true, true>(d, ctl, gtid(), gstride());
    else dense_arena_body<true>(d, ctl, gtid(), gstride());
  }
}

// The buffered children's dense slots in a launch of their own (the TOPK
// leaf path, and the levels below M).
template <bool LEVEL_M>
__global__ void __launch_bounds__(kThreads) k_dense_arena(Dev d) {
  pdl_enter();
  Ctl* ctl = d.ctl;
  if (no_copy(ctl) || ctl->skip_dense) return;
  dense_arena_body<LEVEL_M>(d, ctl, gtid(), gstride());
}

// Output offsets of every child span; a slot no child filled means a child
// was repeated elsewhere.
struct DenseScan {
  const uint4* dense;
  u64* dst;
  Ctl* ctlp;
  // without levels below M handing spans up, the total is the batch's
  // payload, checked here against the ring (else k_check2 does it)
  bool check_payload;
  u64 out_payload;
  bool split = false;  // split placement: stands down on the errors raised before the fork
  __device__ u64 size(const Ctl* ctl) const {
    if (split) return (ctl->skip_dense || ctl->pre_err) ? 0 : ctl->leaf_dense_total;
    return (ctl->skip_dense || ctl->batch_err) ? 0 : ctl->dense_total + ctl->chain_total;
  }
  __device__ u64 value(u64 j) const {
    uint4 v = dense[j];
    if (v.x != ctlp->epoch) {
      raise_err(ctlp, ALTO_EDUP);
      return 0;
    }
    return v.y;
  }
  __device__ void out(u64 j, u64 excl, u64) const { dst[j] = excl; }
  __device__ void total(Ctl* ctl, u64 t) const {
    dst[size(ctl)] = t;
    ctl->pay_total = t;
    if (check_payload && !halted(ctl) && !ctl->skip_dense && ctl->pay_count + t > out_payload) {
      raise_err(ctl, ALTO_ENOSPC);
      ctl->skip_dense = 1;
    }
  }
};

// The payload against the ring when levels below M hand spans up: level M's
// spans come first, the slots after them are not emitted.
__global__ void k_check2(Dev d) {
  pdl_enter();
  Ctl* ctl = d.ctl;
  if (poisoned(ctl) || ctl->skip_dense) return;
  // level M's spans come first; the slots after them are handed up, not emitted
  if (ctl->chain_total && !ctl->batch_err) ctl->pay_total = d.sc.dst[ctl->dense_total];
  if (ctl->pay_count + ctl->pay_total > d.cfg.out_payload) {
    raise_err(ctl, ALTO_ENOSPC);
    ctl->skip_dense = 1;
  }
}

__device__ __forceinline__ int32_t span_load(const Dev& d, const Batch& b, u32 owner, u32 pos,
                                             u32 k) {
  if (owner == kNone) return b.pay[(u64)pos + k];
  bool ok;
  const u64 a = vec_addr(d.tab, owner, 1, (u64)pos + k, &ok);
  return ok ? d.ar.pool[a] : 0;
}

// Copy every child span into the output payload ring.
//
// Eight lanes take one span (a warp four spans at a time): lane `sub` of the
// group copies elements sub, sub+8, ..., with the first 64 elements' loads
// all issued, as plain predicated loads, before the stores.  With spans of a
// few dozen elements read in an order unrelated to their source order, this
// keeps about as many loads in flight as the memory system can overlap;
// wider groups (16 or 32 lanes a span), narrower ones, more spans per group,
// staging through shared memory (with 16-byte vector loads or with bulk
// copies) and scattering in source order instead all measured slower on span
// streams of this shape, and so did a first pass with a per-element fallback
// branch (the loads no longer overlap).  An arena span is read through its
// first chunk; elements past that chunk (a span across a chunk boundary)
// look up their chunk one by one, after the rest.
constexpr int kSpanLanes = 8;
constexpr int kSpanFirst = 8;  // elements per lane in the first pass

// 32 registers: eight blocks per SM, the grid is one wave
template <bool G>
__global__ void __launch_bounds__(kThreads, 8) k_gather(Dev d, Batch bv) {
  pdl_enter();
  const Batch b = batch_of<G>(bv, d);
  Ctl* ctl = d.ctl;
  if (stand_down(d, ctl) || ctl->skip_dense) return;
  const int lane = threadIdx.x & 31, sub = lane % kSpanLanes, grp = lane / kSpanLanes;
  constexpr int kGroups = 32 / kSpanLanes;
  const u32 ep = ctl->epoch;
  const u64 total = d.split ? ctl->leaf_dense_total : ctl->dense_total;
  const u64 base = ctl->pay_base;
  const u64 cap = d.cfg.out_payload;
  int32_t* __restrict__ out = d.out_pay;
  const u64 gw = gtid() >> 5, nw = gstride() >> 5;
  for (u64 jb = gw * kGroups; jb < total; jb += nw * kGroups) {
    const u64 j = jb + grp;
    u32 len = 0, owner = kNone, pos = 0, n1 = 0;
    u64 o = 0;
    const int32_t* src = b.pay;
    if (j < total) {
      const uint4 v = d.sc.dense[j];
      o = base + d.sc.dst[j];
      bool good = v.x == ep && o + v.y <= cap;
      if (good && v.z == kNone) good = (u64)v.w + v.y <= b.n_payload;
      if (good && v.z != kNone)
        good = v.z <= d.tab.mask && (u64)v.w + v.y <= d.tab.vec_n[2 * (u64)v.z + 1];
      if (good) {
        len = v.y;
        owner = v.z;
        pos = v.w;
        if (owner == kNone) {
          src = b.pay + pos;
          n1 = len;
        } else if (len) {
          const int jc = chunk_of(pos);
          const u32 cb = (jc < kNumChunks) ? d.tab.dir[((u64)owner * kVecs + 1) * kNumChunks + jc] : kNone;
          if (cb != kNone) {
            src = d.ar.pool + cb + ((u64)pos - chunk_start(jc));
            const u64 room = chunk_start(jc) + chunk_size(jc) - pos;
            n1 = (room < len) ? (u32)room : len;
          }
        }
      }
    }
    int32_t val[kSpanFirst];
#pragma unroll
    for (int q = 0; q < kSpanFirst; ++q) {
      const u32 k = sub + kSpanLanes * q;
      val[q] = (k < n1) ? src[k] : 0;
    }
#pragma unroll
    for (int q = 0; q < kSpanFirst; ++q) {
      const u32 k = sub + kSpanLanes * q;
      if (k < n1) out[o + k] = val[q];
    }
    for (u32 k = kSpanLanes * kSpanFirst + sub; k < n1; k += kSpanLanes) out[o + k] = src[k];
    for (u32 k = n1 + sub; k < len; k += kSpanLanes) out[o + k] = span_load(d, b, owner, pos, k);
  }
}

// Level l (M < l): the concatenations of its groups completing in this batch,
// copied into the spans they reserved in their parents' payload vectors.  The
// done list holds levels in non-increasing order (levels finalise bottom-up),
// so the level's groups, and their dense slots, form one range.  A warp takes
// 32 consecutive slots; each lane finds its slot's group by binary search,
// then the warp copies the spans one after another.
template <bool G>
__global__ void __launch_bounds__(kThreads) k_chain_gather(Dev d, Batch bv, int l) {
  pdl_enter();
  const Batch b = batch_of<G>(bv, d);
  Ctl* ctl = d.ctl;
  if (no_copy(ctl) || ctl->skip_dense) return;
  const u32 ep = ctl->epoch;
  const u32 nd = min(ctl->n_done, d.sc.done_cap);
  const u32* lvl = d.sc.done_lvl;
  // [x0, x1): done indices of level l
  u32 x0 = 0, x1 = nd;
  {
    u32 lo = 0, hi = nd;  // first index with level <= l
    while (lo < hi) {
      const u32 mid = (lo + hi) >> 1;
      if ((int)lvl[mid] > l) lo = mid + 1;
      else hi = mid;
    }
    x0 = lo;
    hi = nd;  // first index with level < l
    while (lo < hi) {
      const u32 mid = (lo + hi) >> 1;
      if ((int)lvl[mid] >= l) lo = mid + 1;
      else hi = mid;
    }
    x1 = lo;
  }
  if (x0 >= x1) return;
  const u64 j0 = d.sc.c_dense_base[x0], j1 = d.sc.c_dense_base[x1];
  const int lane = threadIdx.x & 31;
  const u64 gw = gtid() >> 5, nw = gstride() >> 5;
  for (u64 jb = j0 + gw * 32; jb < j1; jb += nw * 32) {
    const u64 j = jb + lane;
    u32 len = 0, owner = kNone, pos = 0, P = 0;
    u64 dp = 0;
    if (j < j1 && j < d.cfg.dense_cap) {
      u32 lo = x0, hi = x1;  // last index with slot base <= j
      while (hi - lo > 1) {
        const u32 mid = (lo + hi) >> 1;
        if (d.sc.c_dense_base[mid] <= j) lo = mid;
        else hi = mid;
      }
      const u32 e = d.sc.done_e[lo] & d.tab.mask;
      const uint4 v = d.sc.dense[j];
      const u32 par = d.tab.par[e] & d.tab.mask;
      const u64 to = (d.tab.app[e] & kPos40) + (d.sc.dst[j] - d.sc.dst[d.sc.c_dense_base[lo]]);
      bool good = v.x == ep && to + v.y <= d.tab.vec_n[2 * (u64)par + 1];
      if (good && v.z == kNone) good = (u64)v.w + v.y <= b.n_payload;
      if (good && v.z != kNone)
        good = v.z <= d.tab.mask && (u64)v.w + v.y <= d.tab.vec_n[2 * (u64)v.z + 1];
      if (good) {
        len = v.y;
        owner = v.z;
        pos = v.w;
        P = par;
        dp = to;
      }
    }
    const u32 cnt = (j1 - jb < 32) ? (u32)(j1 - jb) : 32u;
    for (u32 k = 0; k < cnt; ++k) {
      const u32 Lk = __shfl_sync(0xFFFFFFFFu, len, k);
      if (Lk == 0) continue;
      const u32 ow = __shfl_sync(0xFFFFFFFFu, owner, k);
      const u32 ps = __shfl_sync(0xFFFFFFFFu, pos, k);
      const u32 Pk = __shfl_sync(0xFFFFFFFFu, P, k);
      const u64 dk = __shfl_sync(0xFFFFFFFFu, dp, k);
      for (u32 q = lane; q < Lk; q += 32) {
        const int32_t val = span_load(d, b, ow, ps, q);
        bool ok;
        const u64 a = vec_addr(d.tab, Pk, 1, dk + q, &ok);
        if (ok) d.ar.pool[a] = val;
      }
    }
  }
}

// Streaming release, after the gather has copied the released spans out:
// drop the released children (those below rnew) of entry e from its buffer.
// The kept meta entries and payload spans move down in place, in their order
// (a destination never lies above its source, and the warp reads each step's
// 32 entries, or 32 elements, before it writes them); chunks of classes past
// the new sizes go back to the free stacks.  All 32 lanes call it together;
// returns the elements freed (lanes 0 and 1).
__device__ u64 compact_buffer(const Dev& d, Ctl* ctl, u32 e) {
  const int lane = threadIdx.x & 31;
  const u32 r1 = d.tab.rnew[e];
  const u32 m = d.tab.vec_n[2 * (u64)e], p = d.tab.vec_n[2 * (u64)e + 1];
  u32 km = 0, kp = 0;  // kept entries and elements so far
  for (u32 kb = 0; kb < m; kb += 32) {
    const u32 k = kb + lane;
    u32 c = 0, pos = 0, end = 0;
    bool ok = false;
    if (k < m) {
      bool ok0, ok1 = true;
      const u64 a = vec_addr(d.tab, e, 0, 2 * (u64)k, &ok0);
      if (ok0) {
        c = (u32)d.ar.pool[a];
        pos = (u32)d.ar.pool[a + 1];
      }
      if (k + 1 < m) {
        const u64 a2 = vec_addr(d.tab, e, 0, 2 * (u64)(k + 1) + 1, &ok1);
        end = ok1 ? (u32)d.ar.pool[a2] : pos;
      } else {
        end = p;
      }
      ok = ok0 && ok1 && end >= pos && end <= p;
    }
    const bool keep = ok && c >= r1;
    const u32 len = keep ? end - pos : 0u;
    u32 incl = len;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const u32 y = __shfl_up_sync(0xFFFFFFFFu, incl, o);
      if (lane >= o) incl += y;
    }
    const u32 kmask = __ballot_sync(0xFFFFFFFFu, keep);
    const u32 nidx = km + __popc(kmask & lanemask_lt());
    const u32 npos = kp + incl - len;
    __syncwarp();  // every lane has read this step's entries
    if (keep) {
      bool okw;
      const u64 a = vec_addr(d.tab, e, 0, 2 * (u64)nidx, &okw);
      if (okw) {
        d.ar.pool[a] = (int32_t)c;
        d.ar.pool[a + 1] = (int32_t)npos;
      }
    }
    // the kept spans, one after another, 32 elements a step
    u32 pend = kmask;
    while (pend) {
      const int src = __ffs(pend) - 1;
      pend &= pend - 1;
      const u32 sp = __shfl_sync(0xFFFFFFFFu, pos, src);
      const u32 dp = __shfl_sync(0xFFFFFFFFu, npos, src);
      const u32 sl = __shfl_sync(0xFFFFFFFFu, len, src);
      if (sp == dp) continue;
      for (u32 q0 = 0; q0 < sl; q0 += 32) {
        const u32 q = q0 + lane;
        int32_t v = 0;
        bool okr = false;
        if (q < sl) {
          const u64 a = vec_addr(d.tab, e, 1, (u64)sp + q, &okr);
          if (okr) v = d.ar.pool[a];
        }
        __syncwarp();
        if (okr) {
          bool okw;
          const u64 a = vec_addr(d.tab, e, 1, (u64)dp + q, &okw);
          if (okw) d.ar.pool[a] = v;
        }
        __syncwarp();
      }
    }
    km += __popc(kmask);
    kp += __shfl_sync(0xFFFFFFFFu, incl, 31);
  }
  u64 freed = 0;
  if (lane < kVecs) {
    const int vec = lane;
    const u64 old_el = (vec == 0) ? 2 * (u64)m : (u64)p;
    const u64 new_el = (vec == 0) ? 2 * (u64)km : (u64)kp;
    if (old_el > new_el) {
      const int jf = (new_el == 0) ? 0 : chunk_of(new_el - 1) + 1;
      const int jl = min(chunk_of(old_el - 1), kNumChunks - 1);
      for (int j = jf; j <= jl; ++j) {
        u32* slot = &d.tab.dir[((u64)e * kVecs + vec) * kNumChunks + j];
        if (*slot != kNone) {
          free_chunk(d.ar, ctl, j, *slot);
          freed += chunk_size(j);
        }
        *slot = kNone;
      }
    }
  }
  __syncwarp();
  if (lane == 0) {
    d.tab.vec_n[2 * (u64)e] = km;
    d.tab.vec_n[2 * (u64)e + 1] = kp;
    // a group above the leaf parent takes its children's spans at its cursor
    if (d.cfg.concat_level < d.cfg.depth - 1) d.tab.cur[e] = ((u64)km << 40) | kp;
  }
  return freed;
}

// One warp per partial release that took children buffered by earlier batches.
__global__ void __launch_bounds__(kThreads) k_stream_compact(Dev d) {
  pdl_enter();
  Ctl* ctl = d.ctl;
  if (no_copy(ctl) || ctl->skip_dense) return;
  const int lane = threadIdx.x & 31;
  const u32 nd = min(ctl->n_done, d.sc.done_cap);
  const u32 gw = gtid() >> 5, nw = gstride() >> 5;
  u64 freed = 0;
  for (u32 db = gw * 32; db < nd; db += nw * 32) {
    u32 todo = __ballot_sync(0xFFFFFFFFu, db + lane < nd && d.sc.done_part[db + lane] == 2u);
    while (todo) {
      const u32 di = db + (u32)(__ffs(todo) - 1);
      todo &= todo - 1;
      freed += compact_buffer(d, ctl, d.sc.done_e[di] & d.tab.mask);
    }
  }
  if (freed) atomicAdd((unsigned long long*)&ctl->arena_used, (unsigned long long)(-(long long)freed));
}

__global__ void __launch_bounds__(kThreads) k_records(Dev d) {
  pdl_enter();
  Ctl* ctl = d.ctl;
  if (poisoned(ctl)) return;
  __shared__ u32 s_del;
  __shared__ unsigned long long s_freed;
  __shared__ u32 s_cnt[kNumChunks];
  __shared__ u32 s_rank[kNumChunks];
  __shared__ int s_base[kNumChunks];
  if (threadIdx.x == 0) {
    s_del = 0;
    s_freed = 0;
  }
  const int M = d.cfg.concat_level;
  const u32 nd = min(ctl->n_done, d.sc.done_cap);
  const bool skip = ctl->skip_dense || ctl->skip_rec;
  for (u32 base = blockIdx.x * blockDim.x; base < nd; base += gridDim.x * blockDim.x) {
    if (threadIdx.x < kNumChunks) {
      s_cnt[threadIdx.x] = 0;
      s_rank[threadIdx.x] = 0;
    }
    __syncthreads();
    const u32 di = base + threadIdx.x;
    const bool mine = di < nd;
    u32 e = 0;
    int l = 0;
    u64 el[kVecs] = {0, 0};
    bool part = false;  // a partial release: the group stays open
    if (mine) {
      e = d.sc.done_e[di] & d.tab.mask;
      l = (int)d.sc.done_lvl[di];
      const u32 cs = d.sc.done_cseq[di];
      const u32 r = d.sc.done_rank[di];
      if (cs < d.cfg.n_max) {
        d.sc.mask[cs] = 0;
        d.sc.mblk[cs >> 5] = 0;
      }
      if (d.cfg.stream) {
        part = d.sc.done_part[di] != 0;
        d.sc.done_part[di] = 0;
        if (part) d.tab.rel[e] = d.tab.rnew[e];  // the group goes on from the end of this release
      }
      if (!skip && r != kNone) {
        alto_record rec;
        rec.completion_seq = ctl->seq_base + cs;
        if (M >= 0) {
          const u64 db = min(d.sc.r_dense_base[r], ctl->dense_total);
          const u64 de = min(db + d.sc.r_dense_n[r], ctl->dense_total);
          rec.payload_off = ctl->pay_count + d.sc.dst[db];
          rec.payload_len = (l == M) ? d.sc.dst[de] - d.sc.dst[db] : 0;
        } else {
          rec.payload_off = ctl->pay_count;
          rec.payload_len = 0;
        }
        u32 tn = d.sc.r_topk_n[r];
        const u64 to = ctl->topk_count + d.sc.r_topk_off[r];
        if (to + tn > d.cfg.out_topk) tn = 0;
        rec.topk_off = to;
        rec.topk_n = (uint16_t)tn;
        rec.parent_id = (u32)d.tab.key[e];
        rec.n_children = part ? d.tab.rnew[e] : d.tab.hot[e].last + 1;
        rec.level = (uint8_t)l;
        rec.ops = part ? (uint8_t)(ALTO_PAYLOAD_CONCAT | ALTO_OPS_PARTIAL)
                       : (uint8_t)(((l == M) ? 1 : 0) | (d.cfg.score_op[l] << 2));
        rec.score = (!part && d.cfg.score_op[l] != ALTO_SCORE_NONE) ? key_score(d.tab.hot[e].smax) : 0.0f;
        d.out_rec[ctl->rec_count + r] = rec;
        for (u32 q = 0; q < tn; ++q) {
          const u64 v = d.tab.topk[(u64)e * d.tab.kk + q];
          alto_topk_pair p;
          p.child_index = ~(u32)v;
          p.score = key_score((u32)(v >> 32));
          d.out_topk[to + q] = p;
        }
      }
      if (M >= 0 && l >= M && !part) {
        for (int vec = 0; vec < kVecs; ++vec) {
          el[vec] = (u64)d.tab.vec_n[2 * (u64)e + vec] * (vec == 0 ? 2 : 1);
          if (el[vec] == 0) continue;
          const int jl = min(chunk_of(el[vec] - 1), kNumChunks - 1);
          for (int j = 0; j <= jl; ++j) atomicAdd(&s_cnt[j], 1u);
        }
      }
      if (!part) {
        d.tab.ready[e] = 0;
        d.tab.key[e] = kTomb;
        d.tab.cur[e] = 0;  // a slot taken later may receive spans in the launch that inserts it
        atomicAdd(&s_del, 1u);
      }
    }
    __syncthreads();
    // one push per chunk class for the whole block
    if (threadIdx.x < kNumChunks && s_cnt[threadIdx.x]) {
      const int j = threadIdx.x;
      s_base[j] = atomicAdd(&ctl->top[j], (int)s_cnt[j]);
      atomicAdd(&s_freed, (unsigned long long)s_cnt[j] * chunk_size(j));
    }
    __syncthreads();
    if (mine && M >= 0 && l >= M && !part) {
      for (int vec = 0; vec < kVecs; ++vec) {
        if (el[vec] == 0) continue;
        const int jl = min(chunk_of(el[vec] - 1), kNumChunks - 1);
        for (int j = 0; j <= jl; ++j) {
          const u32 chunk = d.tab.dir[((u64)e * kVecs + vec) * kNumChunks + j];
          const u64 pos = (u64)s_base[j] + atomicAdd(&s_rank[j], 1u);
          if (chunk != kNone && pos < d.ar.stack_cap[j]) d.ar.stack[d.ar.stack_off[j] + pos] = chunk;
        }
      }
    }
    __syncthreads();
  }
  if (threadIdx.x == 0) {
    if (s_del) atomicAdd((unsigned long long*)&ctl->live_groups, (unsigned long long)(-(long long)s_del));
    if (s_freed) atomicAdd((unsigned long long*)&ctl->arena_used, (unsigned long long)(-(long long)s_freed));
  }
}

// End of a batch: latch its error, or count its output into the ring.
__device__ void end_batch(Ctl* ctl) {
  if (ctl->status != ALTO_OK) return;
  if (ctl->batch_err) {
    ctl->status = -(ctl->batch_err & 0xFF);
    return;
  }
  ctl->rec_count += ctl->n_done;
  ctl->pay_count += ctl->pay_total;
  ctl->topk_count += ctl->topk_total;
  ctl->seq_base += ctl->n;
}

// Turn deleted slots back into free ones where no probe chain runs through
// them: a tombstone followed (after more tombstones) by a free slot.  The
// batch's records are written by now, so thread 0 also ends the batch (the
// kernel is the last of a push).
__global__ void __launch_bounds__(kThreads) k_sweep(Dev d) {
  pdl_enter();
  Ctl* ctl = d.ctl;
  if (blockIdx.x == 0 && threadIdx.x == 0) end_batch(ctl);
  if (poisoned(ctl)) return;
  const u32 nd = min(ctl->n_done, d.sc.done_cap);
  const u32 mask = d.tab.mask;
  volatile u64* key = d.tab.key;
  for (u32 di = gtid(); di < nd; di += gstride()) {
    const u32 e = d.sc.done_e[di];
    if (key[e] != kTomb) continue;
    u32 p = (e + 1) & mask;
    int steps = 0;
    while (key[p] == kTomb && steps < d.tab.max_probe) {
      p = (p + 1) & mask;
      ++steps;
    }
    if (key[p] != kEmpty) continue;
    key[e] = kEmpty;
    u32 q = (e - 1) & mask;
    steps = 0;
    while (key[q] == kTomb && steps < d.tab.max_probe) {
      key[q] = kEmpty;
      q = (q - 1) & mask;
      ++steps;
    }
  }
}

__global__ void k_end(Ctl* ctl) {
  pdl_enter();
  end_batch(ctl);
}

}  // namespace alto

using namespace alto;

// ---------------------------------------------------------------------------
// host side
// ---------------------------------------------------------------------------
struct alto_agg {
  alto_agg_config cfg;
  alto_allocator alloc;
  bool use_async;
  int device;
  int num_sms;
  int tbits;
  Dev d;
  SortBuffers leaf_sort, up_sort;
  LookbackState lbs;
  Ctl* h_ctl;  // pinned host copy for drain
  std::vector<void*> blocks;
  u64 pushed;    // batches pushed, empty ones included
  u64 launched;  // batches that launched work (the device's batch epochs)
  u64 drain_first;
  int latched;
  // output rings: [1] is allocated only with ALTO_FLAG_DOUBLE_RING; pushes
  // write ring [ring_cur], and a drain hands it out and moves to the other
  alto_record* ring_rec[2];
  int32_t* ring_pay[2];
  alto_topk_pair* ring_topk[2];
  int ring_cur;
  // measurement hooks
  bool profiling;
  int profile_mode;  // ALTO_PROFILE_STAGES or ALTO_PROFILE_HOT
  cudaStream_t last_stream;
  int64_t prof_pushes;
  int64_t launches;
  double stage_ms[ALTO_NUM_STAGES];
  int64_t stage_launches[ALTO_NUM_STAGES];
  std::vector<cudaEvent_t> ev_free;                   // reusable events
  std::vector<std::vector<cudaEvent_t>> ev_pending;  // per push: stage boundaries
  // Pushes of up to kGraphMaxBatch fragments replay a CUDA graph of the
  // push's launch sequence, captured once per (output ring, profiling mode):
  // one launch from the host instead of twenty-odd.  Only the first node's
  // parameters (the batch) and, when profiling, the events of the
  // event-record nodes change from push to push.
  struct PushGraph {
    cudaGraph_t graph = nullptr;
    cudaGraphExec_t exec = nullptr;
    cudaGraphNode_t begin = nullptr;                 // k_begin
    std::vector<cudaGraphNode_t> ev_node;            // per stage boundary (null: none)
    int64_t launches = 0;                            // kernels of one replay
    int64_t stage_launches[ALTO_NUM_STAGES] = {};
    bool failed = false;                             // capture failed: launch directly
  };
  PushGraph graphs[2][3][4];  // [ring][profiling: off, stages, hot][batch size class]
  cudaStream_t cap_stream = nullptr;
  // direct launches: the side streams (records and sweep beside the gather;
  // with a split placement the leaf parents' payload path and the arena
  // copies) and their events
  cudaStream_t side = nullptr, side3 = nullptr;
  cudaEvent_t ev_fork = nullptr, ev_join = nullptr, ev_dense = nullptr, ev_join3 = nullptr;
  LookbackState lbs2{};                 // the split placement's look-back state
  std::vector<cudaEvent_t> cap_events;  // recorded at capture only (the graphs' templates hold them)
  bool direct_only = false;   // ALTO_FLAG_DIRECT_LAUNCH
  bool reset_pending = false; // a drain handed out the ring: the next push resets its counters
};

namespace {

// Stage boundaries of one push, recorded when profiling is on.
struct StageClock {
  alto_agg* h;
  cudaStream_t s;
  std::vector<cudaEvent_t> ev;
  int stage = 0;
  int launches_at_start = 0;
  bool capturing = false;
  StageClock(alto_agg* h_, cudaStream_t s_) : h(h_), s(s_) {}
  cudaEvent_t take() {
    cudaEvent_t e;
    if (!h->ev_free.empty()) {
      e = h->ev_free.back();
      h->ev_free.pop_back();
    } else if (cudaEventCreate(&e) != cudaSuccess) {
      return nullptr;
    }
    return e;
  }
  // mark the start of stage `st` (stages must be entered in order); in the hot
  // mode only the boundaries around the leaf accumulate and the gather get an
  // event
  void enter(int st, cudaStream_t on = nullptr) {
    if (!h->profiling) return;
    if (!on) on = s;
    while ((int)ev.size() <= st) {
      const int bnd = (int)ev.size();
      cudaEvent_t e = nullptr;
      if (h->profile_mode == ALTO_PROFILE_STAGES || bnd == 2 || bnd == 3 || bnd == 8 || bnd == 9) {
        e = take();
        // inside a stream capture only an external record becomes an
        // event-record node (a plain one just orders captured streams)
        if (e) {
          if (capturing) cudaEventRecordWithFlags(e, on, cudaEventRecordExternal);
          else cudaEventRecord(e, on);
        }
      }
      ev.push_back(e);
    }
  }
};

void collect_profile(alto_agg* h) {
  for (auto& ev : h->ev_pending) {
    for (int st = 0; st < ALTO_NUM_STAGES && st + 1 < (int)ev.size(); ++st) {
      float ms = 0.0f;
      if (ev[st] && ev[st + 1] && cudaEventElapsedTime(&ms, ev[st], ev[st + 1]) == cudaSuccess)
        h->stage_ms[st] += ms;
    }
    for (cudaEvent_t e : ev)
      if (e) h->ev_free.push_back(e);
  }
  h->ev_pending.clear();
}

LookbackState lb_region(const LookbackState& lb, int k) {
  LookbackState r = lb;
  r.desc += (u64)k * lb.tiles;
  return r;
}

template <class F, class L>
void launch_scan3(const LookbackState& lb, Ctl* ctl, const F& f0, const F& f1,
                  const F& f2, u64 cap, int site, u64 spin, cudaStream_t s, const L& last) {
  u64 tiles = (cap + kScanTile - 1) / kScanTile;
  if (tiles == 0) tiles = 1;
  // the record scans run over completed groups (far fewer than fragments):
  // a small persistent grid, so that hundreds of idle CTAs do not contend on
  // the tile and exit counters
  dim3 grid((unsigned)std::min<u64>(tiles, 32), 3);
  launch_pdl(k_scan3<F, L>, grid, kScanThreads, 0, s, f0, f1, f2, lb_region(lb, 0), lb_region(lb, 1),
             lb_region(lb, 2), ctl, site, spin, last);
}

template <class F>
void launch_scan(const LookbackState& lb, int num_sms, Ctl* ctl, const F& f, u64 cap, int site,
                 u64 spin, cudaStream_t s, int max_grid = 0) {
  u64 tiles = (cap + kScanTile - 1) / kScanTile;
  if (tiles == 0) tiles = 1;
  // up to four CTAs per SM: with a functor that loads and stores per element
  // the extra CTAs hide its latency (one per SM was faster only for a bare
  // sum in isolation)
  int grid = (int)std::min<u64>(tiles, (u64)num_sms * 4);
  if (max_grid > 0) grid = std::min(grid, max_grid);
  launch_pdl(k_scan<F>, grid, kScanThreads, 0, s, f, lb, ctl, site, &ctl->exit_ctr[site], spin);
}

// What one batch enqueues after k_begin, for the handle's push and for the
// one-shot entry point alike (its last kernel, k_sweep, also ends the batch).  `stage` (may be null) marks the
// start of each profiling stage; `launches` counts the kernels.
struct Pipeline {
  Dev d;
  SortBuffers* leaf_sort;
  SortBuffers* up_sort;
  LookbackState lbs;
  int num_sms;
  int tbits;
  u32 nmax;
  // fragments of the largest batch these launches serve (nmax for a direct
  // launch, the size class of a captured graph): grids of kernels whose work
  // the batch size bounds are sized for it
  u32 nb;
  cudaStream_t s;
  void (*stage)(void* ctx, int st, int64_t launches) = nullptr;
  void* stage_ctx = nullptr;
  // a second stream (with its fork and join events) on which the records and
  // the table sweep run beside the payload gather, or, with a split
  // placement, the completing leaf parents' payload path; null: one stream
  cudaStream_t s2 = nullptr;
  cudaEvent_t ev_fork = nullptr, ev_join = nullptr;
  // split placement: a third stream for the open groups' arena copies, the
  // second stream's look-back state, and the events after its length scan
  // and at the end of the third stream
  cudaStream_t s3 = nullptr;
  cudaEvent_t ev_dense = nullptr, ev_join3 = nullptr;
  LookbackState lbs2{};
  int64_t launches = 0;
  void (*stage_on)(void* ctx, int st, int64_t launches, cudaStream_t on) = nullptr;
  void enter(int st) {
    if (stage) stage(stage_ctx, st, launches);
  }
  // a stage boundary recorded on another stream (split placement: the gather)
  void enter_on(int st, cudaStream_t on) {
    if (stage_on) stage_on(stage_ctx, st, launches, on);
    else enter(st);
  }
};

// Launch sites of the split placement's scans (its rank scan, three
// record-style scans and its length scan): above every site the main
// stream's scans take (at most 5 + 5 (kMaxDepth - 1) + 4).
constexpr int kSplitSite = kSites - 5;
static_assert(5 + 5 * (kMaxDepth - 1) + 4 <= kSplitSite, "scan launch sites overlap");

// Blocks of 256 threads of `kernel` resident per SM (cached per kernel): a
// grid-stride kernel whose grid is exactly one wave has no ragged tail.
int blocks_per_sm(const void* kernel) {
  static std::mutex mu;
  static std::vector<std::pair<const void*, int>> cache;
  std::lock_guard<std::mutex> lock(mu);
  for (auto& kv : cache)
    if (kv.first == kernel) return kv.second;
  int nb = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&nb, kernel, kThreads, 0) != cudaSuccess || nb < 1)
    nb = 1;
  cache.emplace_back(kernel, nb);
  return nb;
}

template <bool G>
void enqueue_batch(Pipeline& p, const Batch& bt) {
  Dev d = p.d;
  cudaStream_t s = p.s;
  const int D = d.cfg.depth;
  const int M = d.cfg.concat_level;
  const u32 nmax = p.nmax;
  const u32 nb = std::min(p.nb, nmax);
  // a grid of at most `full` blocks, no more than `items` of `per` each need
  // (small batches launch small grids: idle blocks still cost their launch)
  auto fit = [](int full, u64 items, u64 per) {
    const u64 need = std::max<u64>(1, (items + per - 1) / per);
    return (int)std::min<u64>((u64)full, need);
  };
  const bool small = nb < nmax;
  const int grid = fit(p.num_sms * 8, nb, kThreads);    // kernels over fragments or leaves
  const int sgrid = fit(p.num_sms * 2, nb, kThreads);   // kernels over groups (fewer items)
  // kernels over completed groups: a fragment completes at most one a level
  const int dgrid = fit(p.num_sms * 2, (u64)nb * D, kThreads);
  // kernels whose work the batch does not bound (buffered children of the
  // groups it completes, payload): one block an SM for a small batch
  const int ugrid = small ? p.num_sms : p.num_sms * 2;
  bool forked = false;  // records and sweep on the second stream, beside the gather
  // the side stream takes work beside the main one only without streaming
  // release (whose compaction and partial flags order the tail)
  const bool side_ok = p.s2 != nullptr && !d.cfg.stream;
  // streaming release needs each leaf parent's leaves together: the sorted path
  const bool leaf_sorted = d.cfg.score_op[D - 1] == ALTO_SCORE_TOPK || d.cfg.stream_leaf;
  // Split placement (CONCAT at the leaf parent, atomic leaf level): right
  // after the leaf finalize, the open groups' arena copies go to the third
  // stream and the completing leaf parents' payload path (their ranks among
  // themselves and offsets, the placement, the length scan, the gather) to
  // the second, beside the upper levels and the record scans on this one.
  const bool split = side_ok && p.s3 != nullptr && M == D - 1 && !leaf_sorted;
  d.split = split ? 1 : 0;
  // streaming release with the CONCAT level above the leaf parent: right
  // after level M, the releases of its groups left open (see k_up_meta)
  const bool stream_up = d.cfg.stream && !d.cfg.stream_leaf;
  auto up_release = [&](const u32* list, const u32* seg_start) {
    launch_pdl(k_up_meta, dgrid, kThreads, 0, s, d);
    launch_pdl(k_up_release, ugrid, kThreads, 0, s, d, list, seg_start);
    launch_pdl(k_up_rel_seq, dgrid, kThreads, 0, s, d);
    launch_pdl(k_up_rel_mask, dgrid, kThreads, 0, s, d);
    p.launches += 4;
  };
  const u64 spin = d.cfg.spin_limit;
  const u32 dcap = d.sc.done_cap;
  int sl = 0;  // launches inside sort_pairs
  int site = 0;
  launch_pdl(k_ingest<G>, grid, kThreads, 0, s, d, bt);
  p.launches += 1;
  int set = 0;
  // touched entries of consecutive levels, alternately
  u32* lists[2] = {d.sc.up_seg_start, d.sc.up_list2};
  int li = 0;
  if (leaf_sorted) {
    // leaf level with TOPK: sort fragments by their leaf-parent group so that
    // each group's candidates are contiguous for the segmented top-k
    p.enter(1);
    int cur = sort_pairs(&d.ctl->n, nb, p.tbits, true, *p.leaf_sort, d.ctl, site, spin, p.num_sms,
                         s, &sl);
    p.launches += sl;
    sl = 0;
    d.sc.leaf_keys = p.leaf_sort->keys[cur];
    d.sc.leaf_perm = p.leaf_sort->vals[cur];
    p.enter(2);
    SegFind f{d.sc.leaf_keys, d.sc.leaf_seg_start, d.sc.leaf_seg_of, &d.ctl->n, nmax,
              &d.ctl->n_segs[D - 1]};
    launch_scan(p.lbs, p.num_sms, d.ctl, f, nb, site + 4, spin, s);
    launch_pdl(k_reduce<true, G>, fit(p.num_sms * blocks_per_sm((const void*)k_reduce<true, G>), nb, kThreads),
               kThreads, 0, s, d, bt, D - 1, d.sc.leaf_keys, d.sc.leaf_perm, d.sc.leaf_seg_start, set);
    launch_pdl(k_reduce_big<true, G>, fit(p.num_sms, nb, kBigSeg), kBigThreads, 0, s, d, bt, D - 1,
               d.sc.leaf_keys, d.sc.leaf_perm, d.sc.leaf_seg_start, set);
    p.launches += 3;
    if (d.cfg.stream_leaf) {
      launch_pdl(k_reduce_rel<G>, fit(p.num_sms * blocks_per_sm((const void*)k_reduce_rel<G>), nb, 8), kThreads,
                 0, s, d, bt, d.sc.leaf_keys, d.sc.leaf_perm, d.sc.leaf_seg_start, set);
      p.launches += 1;
    }
  } else {
    // leaf level without TOPK: accumulate into the table in arrival order
    // (plain stream order: the measurement hooks time this kernel on its own)
    p.enter(2);
    k_leaf_accumulate<G><<<grid, kThreads, 0, s>>>(d, bt);
    p.enter(3);
    launch_pdl(k_up_finalize<true, G>, sgrid, kThreads, 0, s, d, bt, D - 1, set,
               (const u32*)d.sc.leaf_seg_start, lists[li]);
    p.launches += 2;
    if (split) {
      cudaEventRecord(p.ev_fork, s);
      // the open groups' leaves to the arena
      cudaStreamWaitEvent(p.s3, p.ev_fork, 0);
      launch_pdl(k_leaf_place<G, 1>, grid, kThreads, 0, p.s3, d, bt);
      cudaEventRecord(p.ev_join3, p.s3);
      // the completing leaf parents ranked among themselves, their dense
      // slots and buffered spans by that rank, their placement and the
      // length scan; the records on this stream wait for those
      cudaStreamWaitEvent(p.s2, p.ev_fork, 0);
      LeafRunScan fr{d.sc.lblk, d.sc.lprefix};
      launch_scan(p.lbs2, p.num_sms, d.ctl, fr, nb / 32 + 1, kSplitSite, spin, p.s2);
      launch_pdl(k_leaf_rank, dgrid, kThreads, 0, p.s2, d);
      {
        const u32* nl = &d.ctl->n_done_leaf;
        CountScan l0{d.sc.l_dense_n, d.sc.l_dense_base, nl, dcap, 4};
        CountScan l1{d.sc.l_meta_n, d.sc.l_arena_base, nl, dcap, 5};
        CountScan l2{nullptr, nullptr, nl, 0, 3};
        launch_scan3(p.lbs2, d.ctl, l0, l1, l2, std::min<u64>(dcap, nb), kSplitSite + 1, spin, p.s2,
                     LeafCheck{d.cfg.dense_cap});
      }
      // three quarters of the block slots: the upper levels and the record
      // scans run beside it
      launch_pdl(k_leaf_place<G, 2>, std::min(grid, p.num_sms * 6), kThreads, 0, p.s2, d, bt);
      DenseScan fd{d.sc.dense, d.sc.dst, d.ctl, true, d.cfg.out_payload, true};
      launch_scan(p.lbs2, p.num_sms, d.ctl, fd, d.cfg.dense_cap, kSplitSite + 4, spin, p.s2, small ? 32 : 0);
      cudaEventRecord(p.ev_dense, p.s2);
      // the gather leaves one block slot per SM to the records and the sweep
      int gather_grid = small ? p.num_sms : p.num_sms * blocks_per_sm((const void*)k_gather<G>);
      if (!small) gather_grid -= p.num_sms;
      p.enter_on(8, p.s2);
      k_gather<G><<<gather_grid, kThreads, 0, p.s2>>>(d, bt);
      p.enter_on(9, p.s2);
      cudaEventRecord(p.ev_join, p.s2);
      p.launches += 7;
    }
  }
  site += 5;
  p.enter(4);
  // an atomic finalize looks up the parent groups of the items it emits and,
  // unless the level above is TOPK, adds the items to them as well
  bool looked_up = !leaf_sorted;
  bool added = !leaf_sorted && D >= 2 && d.cfg.score_op[D - 2] != ALTO_SCORE_TOPK;
  for (int l = D - 2; l >= 0; --l) {
    set ^= 1;  // items written by the level below
    if (!looked_up) {
      launch_pdl(k_items_lookup<G>, sgrid, kThreads, 0, s, d, bt, l, set);
      p.launches += 1;
    }
    if (d.cfg.score_op[l] != ALTO_SCORE_TOPK) {
      if (!added) {
        launch_pdl(k_up_accumulate<G>, sgrid, kThreads, 0, s, d, bt, l, set, lists[li]);
        p.launches += 1;
      }
      launch_pdl(k_up_finalize<false, G>, sgrid, kThreads, 0, s, d, bt, l, set, (const u32*)lists[li],
                 lists[li ^ 1]);
      p.launches += 1;
      if (stream_up && l == M) up_release(lists[li], nullptr);
      li ^= 1;
      looked_up = true;
      added = l > 0 && d.cfg.score_op[l - 1] != ALTO_SCORE_TOPK;
      continue;
    }
    looked_up = false;
    added = false;
    int c2 = sort_pairs(&d.ctl->n_segs[l + 1], nb, p.tbits, true, *p.up_sort, d.ctl, site, spin,
                        p.num_sms, s, &sl);
    p.launches += sl;
    sl = 0;
    site += 4;
    d.sc.up_keys = p.up_sort->keys[c2];
    d.sc.up_perm = p.up_sort->vals[c2];
    SegFind f{d.sc.up_keys, d.sc.up_seg_start, nullptr, &d.ctl->n_segs[l + 1], nmax,
              &d.ctl->n_segs[l]};
    launch_scan(p.lbs, p.num_sms, d.ctl, f, nb, site++, spin, s);
    launch_pdl(k_reduce<false, G>, fit(p.num_sms * blocks_per_sm((const void*)k_reduce<false, G>), nb, kThreads),
               kThreads, 0, s, d, bt, l, d.sc.up_keys, d.sc.up_perm, d.sc.up_seg_start, set);
    launch_pdl(k_reduce_big<false, G>, fit(p.num_sms, nb, kBigSeg), kBigThreads, 0, s, d, bt, l, d.sc.up_keys,
               d.sc.up_perm, d.sc.up_seg_start, set);
    p.launches += 3;
    if (stream_up && l == M) up_release(d.sc.up_keys, d.sc.up_seg_start);
  }
  // emission order
  p.enter(5);
  {
    RankScan f{d.sc.mblk, d.sc.prefix, &d.ctl->n};
    launch_scan(p.lbs, p.num_sms, d.ctl, f, nb / 32 + 1, site++, spin, s);
  }
  launch_pdl(k_done_rank, dgrid, kThreads, 0, s, d);
  p.launches += 2;
  const bool chain = M >= 0 && M < D - 1;  // levels below M hand spans up
  {
    CountScan f0{d.sc.r_dense_n, d.sc.r_dense_base, &d.ctl->n_done, dcap, 0,
                 nullptr, nullptr, nullptr, d.tab.mask, nullptr, d.ctl};
    CountScan f1{d.sc.r_topk_n, d.sc.r_topk_off, &d.ctl->n_done, dcap, 1};
    CountScan f2{d.sc.r_meta_n, d.sc.r_arena_base, &d.ctl->n_done, dcap, 2};
    const CapCheck cc{d.cfg.out_records, d.cfg.dense_cap, d.cfg.out_topk, d.sc.done_cap, split};
    const u64 dbound = std::min<u64>(dcap, (u64)nb * D);
    if (chain) launch_scan3(p.lbs, d.ctl, f0, f1, f2, dbound, site, spin, s, NoLast());
    else launch_scan3(p.lbs, d.ctl, f0, f1, f2, dbound, site, spin, s, cc);
    p.launches += 1;
    site += 3;
  }
  if (chain) {
    ChainScan c[3];
    for (int k = 0; k < 3; ++k) {
      c[k].done_e = d.sc.done_e;
      c[k].done_lvl = d.sc.done_lvl;
      c[k].n_dev = &d.ctl->n_done;
      c[k].cap = dcap;
      c[k].which = k;
      c[k].out_off = (k == 1) ? d.sc.c_arena_base : d.sc.c_dense_base;
      c[k].tab = d.tab;
      c[k].arena_pool = d.ar.pool;
      c[k].ctlp = d.ctl;
      c[k].M = M;
      c[k].L = D - 1;
    }
    launch_scan3(p.lbs, d.ctl, c[0], c[1], c[2], std::min<u64>(dcap, (u64)nb * D), site, spin, s,
                 CapCheck{d.cfg.out_records, d.cfg.dense_cap, d.cfg.out_topk, d.sc.done_cap});
    p.launches += 1;
    site += 3;
  }
  if (split) {
    // the records take their payload offsets from the length scan; the
    // sweep ends the batch, so it also waits for the arena copies
    cudaStreamWaitEvent(s, p.ev_dense, 0);
    launch_pdl(k_records, dgrid, kThreads, 0, s, d);
    cudaStreamWaitEvent(s, p.ev_join3, 0);
    launch_pdl(k_sweep, dgrid, kThreads, 0, s, d);
    cudaStreamWaitEvent(s, p.ev_join, 0);
    p.launches += 2;
    p.enter(9);
    return;
  }
  if (M >= 0) {
    p.enter(6);
    if (leaf_sorted) {
      launch_pdl(k_carry_alloc, sgrid, kThreads, 0, s, d);
      launch_pdl(k_fix_tops, 1, 32, 0, s, d.ctl);
      launch_pdl(k_carry_copy<G>, grid, kThreads, 0, s, d, bt);
      p.enter(7);
      launch_pdl(k_dense_batch<G>, grid, kThreads, 0, s, d, bt);
    } else {
      // the leaf finalize already allocated the carried leaves' chunks; the
      // placement also places the children buffered by earlier batches
      p.enter(7);
      launch_pdl(k_leaf_place<G, 3>, grid, kThreads, 0, s, d, bt);
    }
    if (leaf_sorted) launch_pdl(k_dense_arena<true>, ugrid, kThreads, 0, s, d);
    p.launches += leaf_sorted ? 5 : 1;
    if (chain) {
      launch_pdl(k_dense_arena<false>, ugrid, kThreads, 0, s, d);
      p.launches += 1;
    }
    DenseScan fd{d.sc.dense, d.sc.dst, d.ctl, !chain, d.cfg.out_payload};
    launch_scan(p.lbs, p.num_sms, d.ctl, fd, d.cfg.dense_cap, site++, spin, s, small ? 32 : 0);
    p.launches += 1;
    if (chain) {
      launch_pdl(k_check2, 1, 1, 0, s, d);
      p.launches += 1;
    }
    p.enter(8);
    // levels below M hand their concatenations up, deepest first
    for (int l = D - 1; chain && l > M; --l) {
      launch_pdl(k_chain_gather<G>, small ? p.num_sms : p.num_sms * blocks_per_sm((const void*)k_chain_gather<G>),
                 kThreads, 0, s, d, bt, l);
      p.launches += 1;
    }
    // The records and the table sweep touch nothing the gather reads (the
    // gather takes its ring base from pay_base, not from the counters the
    // batch's end moves): with a second stream they run beside it, on one
    // block slot per SM that the gather leaves free.  Not with streaming
    // release (the buffer compaction after the gather reads the partial
    // flags the records clear) or CONCAT above the leaf parent.
    forked = side_ok && M == D - 1;
    int gather_grid = small ? p.num_sms : p.num_sms * blocks_per_sm((const void*)k_gather<G>);
    if (forked) {
      cudaEventRecord(p.ev_fork, s);
      cudaStreamWaitEvent(p.s2, p.ev_fork, 0);
      launch_pdl(k_records, dgrid, kThreads, 0, p.s2, d);
      launch_pdl(k_sweep, dgrid, kThreads, 0, p.s2, d);
      cudaEventRecord(p.ev_join, p.s2);
      p.launches += 2;
      if (!small) gather_grid -= p.num_sms;
    }
    // plain stream order (no programmatic overlap with its neighbours): the
    // gather is the stage the measurement hooks time on their own
    k_gather<G><<<gather_grid, kThreads, 0, s>>>(d, bt);
    p.launches += 1;
  }
  p.enter(9);
  if (forked) {
    cudaStreamWaitEvent(s, p.ev_join, 0);
    return;
  }
  if (d.cfg.stream) {
    // the released spans are out: drop them from the buffers they came from
    launch_pdl(k_stream_compact, ugrid, kThreads, 0, s, d);
    p.launches += 1;
  }
  launch_pdl(k_records, dgrid, kThreads, 0, s, d);
  launch_pdl(k_sweep, dgrid, kThreads, 0, s, d);
  p.launches += 2;
}

void* dev_alloc(alto_agg* h, size_t bytes, cudaStream_t s) {
  bytes = (bytes + 255) & ~(size_t)255;
  if (bytes == 0) bytes = 256;
  void* p = nullptr;
  if (h->use_async) {
    if (cudaMallocAsync(&p, bytes, s) != cudaSuccess) return nullptr;
  } else {
    p = h->alloc.alloc(h->alloc.ctx, bytes, s);
  }
  if (p) h->blocks.push_back(p);
  return p;
}

// Pushes of at most this many fragments replay a captured graph (host
// launch cost matters there); larger ones launch kernel by kernel, whose
// kernels read the batch from their parameters rather than device memory.
// A push replays the graph of the smallest size class that holds it, whose
// grids are sized for that many fragments.
constexpr u32 kGraphMaxBatch = 1u << 17;
constexpr int kGraphClasses = 4;
__host__ __forceinline__ u32 graph_class_bound(int c) { return 1u << (11 + 2 * c); }  // 2K, 8K, 32K, 128K
static_assert(sizeof(alto_agg::graphs[0][0]) / sizeof(alto_agg::PushGraph) == kGraphClasses,
              "one graph per size class");

// Stage bookkeeping of one push's launch sequence: kernels per stage, and the
// stage-boundary events when profiling.
struct PushRec {
  alto_agg* h;
  StageClock clk;
  int stage = 0;
  int64_t l0 = 0;
  int64_t stage_l[ALTO_NUM_STAGES] = {};
  PushRec(alto_agg* h_, cudaStream_t s) : h(h_), clk(h_, s) {}
};

void free_side_streams(alto_agg* h) {
  for (cudaStream_t* x : {&h->side, &h->side3})
    if (*x) cudaStreamDestroy(*x);
  for (cudaEvent_t* x : {&h->ev_fork, &h->ev_join, &h->ev_dense, &h->ev_join3})
    if (*x) cudaEventDestroy(*x);
  h->side = h->side3 = nullptr;
  h->ev_fork = h->ev_join = h->ev_dense = h->ev_join3 = nullptr;
}

// The side streams and their events, made once; false (and none kept) if
// any could not be made: the push then runs on its own stream alone.
bool make_side_streams(alto_agg* h) {
  if (h->side) return true;
  // the second stream carries the split placement's critical path: its
  // blocks go first when blocks of the other streams retire
  int lo_pr = 0, hi_pr = 0;
  if (cudaDeviceGetStreamPriorityRange(&lo_pr, &hi_pr) != cudaSuccess) lo_pr = hi_pr = 0;
  bool ok = cudaStreamCreateWithPriority(&h->side, cudaStreamNonBlocking, hi_pr) == cudaSuccess &&
            cudaStreamCreateWithFlags(&h->side3, cudaStreamNonBlocking) == cudaSuccess;
  for (cudaEvent_t* x : {&h->ev_fork, &h->ev_join, &h->ev_dense, &h->ev_join3})
    ok = ok && cudaEventCreateWithFlags(x, cudaEventDisableTiming) == cudaSuccess;
  if (!ok) free_side_streams(h);
  cudaGetLastError();
  return ok;
}

// The whole launch sequence of one push on stream s: k_begin and the
// pipeline.  G: the kernels read the batch that k_begin stores (graph capture).
// Returns the number of kernels.
template <bool G>
int64_t launch_push(alto_agg* h, cudaStream_t s, const Batch& bt, int reset, PushRec* rec, u32 nb) {
  Dev d = h->d;
  Pipeline p;
  p.d = d;
  p.leaf_sort = &h->leaf_sort;
  p.up_sort = &h->up_sort;
  p.lbs = h->lbs;
  p.num_sms = h->num_sms;
  p.tbits = h->tbits;
  p.nmax = (u32)h->cfg.max_batch_fragments;
  p.nb = nb;
  p.s = s;
  // work beside the main stream goes to the handle's side streams (in a
  // capture they become branches of the graph; not with an event at every
  // stage boundary)
  if (!(h->profiling && h->profile_mode == ALTO_PROFILE_STAGES) && make_side_streams(h)) {
    p.s2 = h->side;
    p.s3 = h->side3;
    p.ev_fork = h->ev_fork;
    p.ev_join = h->ev_join;
    p.ev_dense = h->ev_dense;
    p.ev_join3 = h->ev_join3;
    p.lbs2 = h->lbs2;
  }
  p.stage = [](void* ctx, int st, int64_t launches) {
    PushRec* r = (PushRec*)ctx;
    r->stage_l[r->stage] += launches - r->l0;
    r->l0 = launches;
    r->stage = st;
    r->clk.enter(st);
  };
  p.stage_on = [](void* ctx, int st, int64_t launches, cudaStream_t on) {
    PushRec* r = (PushRec*)ctx;
    r->stage_l[r->stage] += launches - r->l0;
    r->l0 = launches;
    r->stage = st;
    r->clk.enter(st, on);
  };
  p.stage_ctx = rec;
  rec->clk.enter(0);
  launch_pdl(k_begin, 1, 1, 0, s, d.ctl, bt, d.sc.batch, reset);
  p.launches += 1;
  enqueue_batch<G>(p, bt);  // its last kernel also ends the batch
  p.enter(ALTO_NUM_STAGES);
  rec->clk.enter(ALTO_NUM_STAGES);
  return p.launches;
}

// Capture the launch sequence of a push for the handle's current output ring
// and profiling mode, on the handle's own stream (nothing runs), and
// instantiate it.  Every replay sets the parameters of the k_begin node; a
// profiling capture also holds one event-record node per timed stage
// boundary, whose event every replay replaces.  On any failure the graph is marked failed and pushes of that
// kind launch directly.
bool capture_push(alto_agg* h, alto_agg::PushGraph& g, u32 nb) {
  g.failed = true;
  if (!h->cap_stream && cudaStreamCreateWithFlags(&h->cap_stream, cudaStreamNonBlocking) != cudaSuccess) {
    h->cap_stream = nullptr;
    cudaGetLastError();
    return false;
  }

  Batch ph;  // k_begin's parameters of the capture; every replay sets its own
  ph.tags = nullptr;
  ph.off = nullptr;
  ph.pay = nullptr;
  ph.score = nullptr;
  ph.n = 0;
  ph.n_payload = 0;
  if (cudaStreamBeginCapture(h->cap_stream, cudaStreamCaptureModeRelaxed) != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  PushRec rec(h, h->cap_stream);
  rec.clk.capturing = true;
  const int64_t launches = launch_push<true>(h, h->cap_stream, ph, 0, &rec, nb);
  for (cudaEvent_t e : rec.clk.ev)
    if (e) h->cap_events.push_back(e);
  cudaGraph_t graph = nullptr;
  if (cudaStreamEndCapture(h->cap_stream, &graph) != cudaSuccess || graph == nullptr) {
    cudaGetLastError();
    if (graph) cudaGraphDestroy(graph);
    return false;
  }
  size_t nn = 0;
  cudaGraphGetNodes(graph, nullptr, &nn);
  std::vector<cudaGraphNode_t> nodes(nn);
  if (nn) cudaGraphGetNodes(graph, nodes.data(), &nn);
  cudaGraphNode_t begin = nullptr;
  g.ev_node.assign(rec.clk.ev.size(), nullptr);
  for (cudaGraphNode_t nd : nodes) {
    cudaGraphNodeType ty;
    if (cudaGraphNodeGetType(nd, &ty) != cudaSuccess) continue;
    if (ty == cudaGraphNodeTypeKernel) {
      cudaKernelNodeParams kp;
      if (cudaGraphKernelNodeGetParams(nd, &kp) == cudaSuccess && kp.func == (void*)k_begin) begin = nd;
    } else if (ty == cudaGraphNodeTypeEventRecord) {
      cudaEvent_t e = nullptr;
      if (cudaGraphEventRecordNodeGetEvent(nd, &e) != cudaSuccess) continue;
      for (size_t b = 0; b < rec.clk.ev.size(); ++b)
        if (rec.clk.ev[b] == e) g.ev_node[b] = nd;
    }
  }
  cudaGetLastError();
  if (begin == nullptr) {
    cudaGraphDestroy(graph);
    return false;
  }
  cudaGraphExec_t exec = nullptr;
  if (cudaGraphInstantiate(&exec, graph, 0) != cudaSuccess || exec == nullptr) {
    cudaGetLastError();
    cudaGraphDestroy(graph);
    return false;
  }
  g.graph = graph;
  g.exec = exec;
  g.begin = begin;
  g.launches = launches;
  for (int i = 0; i < ALTO_NUM_STAGES; ++i) g.stage_launches[i] = rec.stage_l[i];
  g.failed = false;
  return true;
}

void free_graphs(alto_agg* h) {
  for (auto& ring : h->graphs)
    for (auto& row : ring)
      for (auto& g : row) {
        if (g.exec) cudaGraphExecDestroy(g.exec);
        if (g.graph) cudaGraphDestroy(g.graph);
        g = alto_agg::PushGraph();
      }
  for (cudaEvent_t e : h->cap_events) cudaEventDestroy(e);
  h->cap_events.clear();
  if (h->cap_stream) cudaStreamDestroy(h->cap_stream);
  h->cap_stream = nullptr;
  free_side_streams(h);
}

void free_all(alto_agg* h, cudaStream_t s) {
  for (void* p : h->blocks) {
    if (h->use_async) cudaFreeAsync(p, s);
    else h->alloc.free(h->alloc.ctx, p, s);
  }
  h->blocks.clear();
  if (h->h_ctl) cudaFreeHost(h->h_ctl);
  h->h_ctl = nullptr;
}

u64 next_pow2(u64 x) {
  u64 p = 1;
  while (p < x) p <<= 1;
  return p;
}

int ilog2(u64 x) {
  int b = 0;
  while ((1ull << b) < x) ++b;
  return b;
}

alto_status validate(const alto_agg_config* c) {
  if (c->depth < 1 || c->depth > ALTO_MAX_DEPTH) return ALTO_EINVAL;
  int nconcat = 0;
  for (int l = 0; l < c->depth; ++l) {
    if (c->payload_op[l] != ALTO_PAYLOAD_NONE && c->payload_op[l] != ALTO_PAYLOAD_CONCAT)
      return ALTO_EINVAL;
    if (c->payload_op[l] == ALTO_PAYLOAD_CONCAT) ++nconcat;
    if (c->score_op[l] < ALTO_SCORE_NONE || c->score_op[l] > ALTO_SCORE_TOPK) return ALTO_EINVAL;
    if (c->score_op[l] == ALTO_SCORE_TOPK && (c->topk_k[l] < 1 || c->topk_k[l] > ALTO_MAX_TOPK))
      return ALTO_EINVAL;
  }
  if (nconcat > 1) return ALTO_EINVAL;
  if (c->flags & ~(int64_t)(ALTO_FLAG_STREAM_RELEASE | ALTO_FLAG_DOUBLE_RING | ALTO_FLAG_TEST_STALL |
                            ALTO_FLAG_DIRECT_LAUNCH))
    return ALTO_EINVAL;
  // streaming release needs a CONCAT level
  if ((c->flags & ALTO_FLAG_STREAM_RELEASE) && nconcat == 0) return ALTO_EINVAL;
  if (c->max_batch_fragments < 1 || c->max_batch_fragments >= (1ll << 30)) return ALTO_EINVAL;
  if (c->max_batch_payload < 0 || c->max_batch_payload >= (1ll << 32)) return ALTO_EINVAL;
  if (c->max_open_groups < 0 || c->max_open_groups > (1ll << 25)) return ALTO_EINVAL;
  if (c->arena_elems < 0 || c->arena_elems >= (1ll << 32)) return ALTO_EINVAL;
  if (c->out_records < 0 || c->out_payload_elems < 0 || c->out_topk < 0 || c->max_emit_children < 0 ||
      c->spin_limit < 0)
    return ALTO_EINVAL;
  return ALTO_OK;
}

}  // namespace

extern "C" {

alto_status alto_agg_create(const alto_agg_config* cfg_in, const alto_allocator* alloc, void* stream,
                            alto_agg_t** out) {
  if (cfg_in == nullptr || out == nullptr) return ALTO_EINVAL;
  alto_status v = validate(cfg_in);
  if (v != ALTO_OK) return v;
  if (alloc != nullptr && (alloc->alloc == nullptr || alloc->free == nullptr)) return ALTO_EINVAL;
  alto_agg_config cfg = *cfg_in;
  const u64 nmax = (u64)cfg.max_batch_fragments;
  if (cfg.max_open_groups == 0) cfg.max_open_groups = 1ll << 20;
  if (cfg.arena_elems == 0) cfg.arena_elems = 1ll << 26;
  if (cfg.out_records == 0) cfg.out_records = 4 * (int64_t)nmax;
  if (cfg.out_payload_elems == 0) cfg.out_payload_elems = std::max<int64_t>(4 * cfg.max_batch_payload, 1);
  if (cfg.out_topk == 0) cfg.out_topk = cfg.out_records;
  if (cfg.max_emit_children == 0) cfg.max_emit_children = 4 * (int64_t)nmax;
  if (cfg.spin_limit == 0) cfg.spin_limit = 1ll << 20;

  cudaStream_t s = (cudaStream_t)stream;
  alto_agg* h = new (std::nothrow) alto_agg();
  if (!h) return ALTO_ENOMEM;
  h->cfg = cfg;
  h->use_async = (alloc == nullptr);
  if (alloc) h->alloc = *alloc;
  h->pushed = 0;
  h->launched = 0;
  h->drain_first = 0;
  h->latched = ALTO_OK;
  h->profiling = false;
  h->profile_mode = ALTO_PROFILE_STAGES;
  h->direct_only = (cfg.flags & ALTO_FLAG_DIRECT_LAUNCH) != 0;
  h->last_stream = s;
  h->prof_pushes = 0;
  h->launches = 0;
  for (int i = 0; i < ALTO_NUM_STAGES; ++i) {
    h->stage_ms[i] = 0.0;
    h->stage_launches[i] = 0;
  }
  if (cudaGetDevice(&h->device) != cudaSuccess ||
      cudaDeviceGetAttribute(&h->num_sms, cudaDevAttrMultiProcessorCount, h->device) != cudaSuccess ||
      sort_prepare() != cudaSuccess) {
    delete h;
    return ALTO_ECUDA;
  }
  const int D = cfg.depth;
  int concat = -1, kk = 0;
  bool has_score = false;
  for (int l = 0; l < D; ++l) {
    if (cfg.payload_op[l] == ALTO_PAYLOAD_CONCAT) concat = l;
    if (cfg.score_op[l] != ALTO_SCORE_NONE) has_score = true;
    if (cfg.score_op[l] == ALTO_SCORE_TOPK) kk = std::max(kk, (int)cfg.topk_k[l]);
  }
  const u64 T = next_pow2(std::max<u64>(2 * (u64)cfg.max_open_groups, 1024));
  h->tbits = ilog2(T);
  const u64 done_cap = nmax * (u64)D;
  const u64 dense_cap = (u64)cfg.max_emit_children;
  const u64 PS = next_pow2(std::max<u64>(2 * nmax * (u64)D, 1024));

  Dev& d = h->d;
  memset(&d, 0, sizeof(d));
  bool ok = true;
#define ALLOC(ptr, type, count)                                              \
  do {                                                                       \
    ptr = (type*)dev_alloc(h, sizeof(type) * (size_t)(count), s);            \
    if (!ptr) ok = false;                                                    \
  } while (0)

  ALLOC(d.ctl, Ctl, 1);
  // table
  ALLOC(d.tab.key, u64, T);
  ALLOC(d.tab.hot, Hot, T);
  ALLOC(d.tab.done_idx, u32, T);
  if (concat >= 0) {
    ALLOC(d.tab.vec_n, u32, 2 * T);
    ALLOC(d.tab.dir, u32, T * kVecs * kNumChunks);
  }
  if (kk > 0) ALLOC(d.tab.topk, u64, T * (u64)kk);
  d.tab.chain_len = std::max((D - 1 + 1) & ~1, 2);  // even: read as 16-byte pairs
  ALLOC(d.tab.chain, u64, T * (u64)d.tab.chain_len);
  ALLOC(d.tab.cbits, u64, 4 * T);
  ALLOC(d.tab.cur, u64, T);
  ALLOC(d.tab.dbase, u64, T);
  ALLOC(d.tab.bstate, uint4, T);
  ALLOC(d.tab.ready, u32, T);
  const bool strm = (cfg.flags & ALTO_FLAG_STREAM_RELEASE) != 0;
  if (strm) {
    ALLOC(d.tab.rel, u32, T);
    ALLOC(d.tab.rnew, u32, T);
  }
  d.tab.leaf_level = D - 1;
  d.tab.mask = (u32)(T - 1);
  d.tab.kk = kk;
  d.tab.max_probe = (int)std::min<u64>(T, 1u << 16);
  // arena
  if (concat >= 0) {
    d.ar.elems = (u64)cfg.arena_elems;
    ALLOC(d.ar.pool, int32_t, std::max<u64>(d.ar.elems, 1));
    u64 off = 0;
    for (int j = 0; j < kNumChunks; ++j) {
      d.ar.stack_off[j] = off;
      d.ar.stack_cap[j] = d.ar.elems / (1ull << (kChunk0Log + j)) + 1;
      off += d.ar.stack_cap[j];
    }
    ALLOC(d.ar.stack, u32, off);
  }
  // config
  d.cfg.depth = D;
  d.cfg.concat_level = concat;
  for (int l = 0; l < kMaxDepth; ++l) {
    d.cfg.score_op[l] = (l < D) ? cfg.score_op[l] : 0;
    d.cfg.topk_k[l] = (l < D && cfg.score_op[l] == ALTO_SCORE_TOPK) ? cfg.topk_k[l] : 0;
  }
  d.cfg.has_score = has_score;
  d.cfg.stream = strm;
  d.cfg.stream_leaf = strm && d.cfg.concat_level == D - 1;
  d.cfg.n_max = (u32)nmax;
  d.cfg.out_records = (u64)cfg.out_records;
  d.cfg.out_payload = (u64)cfg.out_payload_elems;
  d.cfg.out_topk = (u64)cfg.out_topk;
  d.cfg.dense_cap = dense_cap;
  d.cfg.spin_limit = (u64)cfg.spin_limit;
  // scratch
  Scratch& sc = d.sc;
  for (int b = 0; b < 2; ++b) {
    ALLOC(h->leaf_sort.keys[b], u32, nmax);
    ALLOC(h->leaf_sort.vals[b], u32, nmax);
    ALLOC(h->up_sort.keys[b], u32, nmax);
    ALLOC(h->up_sort.vals[b], u32, nmax);
  }
  const u64 sort_tiles = nmax / 4096 + 2;
  ALLOC(h->leaf_sort.hist, u32, 4 * 256);
  ALLOC(h->leaf_sort.bin_base, u32, 4 * 256);
  ALLOC(h->leaf_sort.lookback, u64, sort_tiles * 256);
  h->leaf_sort.lb_tiles = sort_tiles;
  h->up_sort.hist = h->leaf_sort.hist;
  h->up_sort.bin_base = h->leaf_sort.bin_base;
  h->up_sort.lookback = h->leaf_sort.lookback;
  h->up_sort.lb_tiles = sort_tiles;
  sc.leaf_sort_keys0 = h->leaf_sort.keys[0];
  sc.up_sort_keys0 = h->up_sort.keys[0];
  ALLOC(sc.leaf_seg_start, u32, nmax + 1);
  ALLOC(sc.leaf_seg_of, u32, nmax);
  ALLOC(sc.up_seg_start, u32, nmax + 1);
  ALLOC(sc.up_list2, u32, nmax);
  for (int b = 0; b < 2; ++b) {
    ALLOC(sc.it_rep[b], u32, nmax);
    ALLOC(sc.it_cseq[b], u32, nmax);
    ALLOC(sc.it_skey[b], u32, nmax);
  }
  ALLOC(sc.seg_vb0, u32, nmax);
  ALLOC(sc.seg_vb1, u32, nmax);
  ALLOC(sc.seg_carry, u32, nmax);
  ALLOC(sc.leaf_pos, u32, nmax);
  ALLOC(sc.mask, u32, (nmax + 31) / 32 * 32);   // whole runs of 32
  ALLOC(sc.mblk, u32, nmax / 32 + 1);
  ALLOC(sc.prefix, u32, nmax);
  ALLOC(sc.done_e, u32, done_cap);
  ALLOC(sc.done_lvl, u32, done_cap);
  ALLOC(sc.done_cseq, u32, done_cap);
  ALLOC(sc.done_rank, u32, done_cap);
  ALLOC(sc.r_done, u32, done_cap);
  ALLOC(sc.r_dense_n, u32, done_cap);
  ALLOC(sc.r_topk_n, u32, done_cap);
  ALLOC(sc.r_meta_n, u32, done_cap);
  ALLOC(sc.r_dense_base, u64, done_cap + 1);
  ALLOC(sc.r_topk_off, u64, done_cap + 1);
  ALLOC(sc.r_arena_base, u64, done_cap + 1);
  if (concat >= 0) {
    ALLOC(sc.dense, uint4, std::max<u64>(dense_cap, 1));
    ALLOC(sc.dst, u64, dense_cap + 1);
  }
  if (concat >= 0 && concat < D - 1) {
    ALLOC(sc.c_dense_base, u64, done_cap + 1);
    ALLOC(sc.c_arena_base, u64, done_cap + 1);
    ALLOC(d.tab.par, u32, T);
    ALLOC(d.tab.cidx, u32, T);
    ALLOC(d.tab.app, u64, T);
  }
  if (concat == D - 1) {
    ALLOC(sc.lblk, u32, nmax / 32 + 1);
    ALLOC(sc.lprefix, u32, nmax / 32 + 1);
    ALLOC(sc.l_done, u32, done_cap);
    ALLOC(sc.l_dense_n, u32, done_cap);
    ALLOC(sc.l_meta_n, u32, done_cap);
    ALLOC(sc.l_dense_base, u64, done_cap + 1);
    ALLOC(sc.l_arena_base, u64, done_cap + 1);
  }
  ALLOC(sc.pairset, u64, PS);
  ALLOC(sc.batch, Batch, 1);
  sc.big_cap = (u32)(nmax / kBigSeg + 1);
  ALLOC(sc.big_seg, u32, (u64)D * sc.big_cap);
  sc.ps_mask = PS - 1;
  sc.done_cap = (u32)done_cap;
  if (strm) {
    // presence bitmaps of one batch: a releasing group takes (candidates / 32 + 1)
    // words, its candidates being the batch's leaves plus its buffered ones
    // (two arena elements of metadata each)
    sc.bm_cap = (nmax + (u64)cfg.arena_elems / 2) / 32 + nmax + 32;
    ALLOC(sc.done_part, u32, done_cap);
    ALLOC(sc.leaf_mrank, u32, nmax);
    ALLOC(sc.bm, u32, sc.bm_cap);
    ALLOC(sc.rel_seg, u32, nmax);
  }
  const u64 scan_tiles = std::max<u64>(std::max<u64>(dense_cap, done_cap), nmax) / kScanTile + 2;
  // three look-back regions for the main stream's scans, three for the
  // split placement's
  ALLOC(h->lbs.desc, ulonglong2, 6 * scan_tiles);
  h->lbs.tiles = scan_tiles;
  h->lbs2.desc = h->lbs.desc ? h->lbs.desc + 3 * scan_tiles : nullptr;
  h->lbs2.tiles = scan_tiles;
  const int rings = (cfg.flags & ALTO_FLAG_DOUBLE_RING) ? 2 : 1;
  for (int r = 0; r < 2; ++r) {
    h->ring_rec[r] = nullptr;
    h->ring_pay[r] = nullptr;
    h->ring_topk[r] = nullptr;
  }
  for (int r = 0; r < rings; ++r) {
    ALLOC(h->ring_rec[r], alto_record, std::max<int64_t>(cfg.out_records, 1));
    ALLOC(h->ring_pay[r], int32_t, std::max<int64_t>(cfg.out_payload_elems, 1));
    ALLOC(h->ring_topk[r], alto_topk_pair, std::max<int64_t>(cfg.out_topk, 1));
  }
  h->ring_cur = 0;
  d.out_rec = h->ring_rec[0];
  d.out_pay = h->ring_pay[0];
  d.out_topk = h->ring_topk[0];
#undef ALLOC
  if (ok && cudaMallocHost((void**)&h->h_ctl, sizeof(Ctl)) != cudaSuccess) {
    h->h_ctl = nullptr;
    ok = false;
  }
  if (!ok) {
    free_all(h, s);
    cudaStreamSynchronize(s);
    delete h;
    return ALTO_ENOMEM;
  }
  // initial state
  cudaMemsetAsync(d.ctl, 0, sizeof(Ctl), s);
  if (cfg.flags & ALTO_FLAG_TEST_STALL) {
    static const int kOne = 1;
    cudaMemcpyAsync(&d.ctl->test_stall, &kOne, sizeof(int), cudaMemcpyHostToDevice, s);
  }
  cudaMemsetAsync(d.tab.key, 0xFF, sizeof(u64) * T, s);
  cudaMemsetAsync(d.tab.ready, 0, sizeof(u32) * T, s);
  launch_pdl(k_init_hot, (int)std::min<u64>((T + kThreads - 1) / kThreads, (u64)h->num_sms * 8), kThreads, 0, s,
             d.tab.hot, T);
  cudaMemsetAsync(d.tab.cur, 0, sizeof(u64) * T, s);
  cudaMemsetAsync(sc.mask, 0, sizeof(u32) * ((nmax + 31) / 32 * 32), s);
  cudaMemsetAsync(sc.mblk, 0, sizeof(u32) * (nmax / 32 + 1), s);
  cudaMemsetAsync(sc.pairset, 0, sizeof(u64) * PS, s);
  cudaMemsetAsync(h->leaf_sort.hist, 0, sizeof(u32) * 4 * 256, s);
  cudaMemsetAsync(h->leaf_sort.lookback, 0, sizeof(u64) * sort_tiles * 256, s);
  cudaMemsetAsync(h->lbs.desc, 0, sizeof(ulonglong2) * 6 * scan_tiles, s);
  if (concat == D - 1) cudaMemsetAsync(sc.lblk, 0, sizeof(u32) * (nmax / 32 + 1), s);
  if (concat >= 0) cudaMemsetAsync(sc.dense, 0, sizeof(uint4) * std::max<u64>(dense_cap, 1), s);
  if (strm) cudaMemsetAsync(sc.done_part, 0, sizeof(u32) * done_cap, s);
  if (cudaGetLastError() != cudaSuccess) {
    free_all(h, s);
    delete h;
    return ALTO_ECUDA;
  }
  *out = h;
  return ALTO_OK;
}

alto_status alto_agg_push_batch(alto_agg_t* h, const alto_batch* b, void* stream) {
  if (h == nullptr || b == nullptr) return ALTO_EINVAL;
  if (h->latched != ALTO_OK) return h->latched;
  const alto_agg_config& cfg = h->cfg;
  if (b->depth != cfg.depth) return ALTO_EINVAL;
  if (b->n < 0 || b->n > cfg.max_batch_fragments) return ALTO_EINVAL;
  if (b->n_payload < 0 || b->n_payload > cfg.max_batch_payload) return ALTO_EINVAL;
  if (b->n > 0 && (b->tags == nullptr || b->payload_off == nullptr)) return ALTO_EINVAL;
  if (b->n_payload > 0 && b->payload == nullptr) return ALTO_EINVAL;
  if (b->n > 0 && h->d.cfg.has_score && b->score == nullptr) return ALTO_EINVAL;
  cudaStream_t s = (cudaStream_t)stream;
  Dev d = h->d;
  const u32 n = (u32)b->n;
  Batch bt;
  bt.tags = b->tags;
  bt.off = b->payload_off;
  bt.pay = b->payload;
  bt.score = h->d.cfg.has_score ? b->score : nullptr;
  bt.n = n;
  bt.n_payload = (u64)b->n_payload;
  if (n == 0) {
    // nothing arrives: no group changes, nothing completes or is released
    h->pushed += 1;
    return ALTO_OK;
  }
  // the pair set's keys carry a 7-bit batch epoch (the device counts batches
  // that launch work): clear it before an epoch value comes round again
  if (h->launched % 127 == 0 && h->launched > 0)
    cudaMemsetAsync(d.sc.pairset, 0, sizeof(u64) * (d.sc.ps_mask + 1), s);
  h->launched += 1;
  h->pushed += 1;
  h->last_stream = s;
  if (h->profiling) h->prof_pushes += 1;
  const int reset = h->reset_pending ? 1 : 0;
  h->reset_pending = false;
  if (!h->direct_only && n <= kGraphMaxBatch) {
    const int pm = !h->profiling ? 0 : (h->profile_mode == ALTO_PROFILE_HOT ? 2 : 1);
    int gc = 0;
    while (gc + 1 < kGraphClasses && n > graph_class_bound(gc)) ++gc;
    alto_agg::PushGraph& g = h->graphs[h->ring_cur][pm][gc];
    if (g.exec == nullptr && !g.failed) capture_push(h, g, graph_class_bound(gc));
    if (g.exec != nullptr) {
      // this push's batch (and counter reset) as k_begin's parameters
      Ctl* ctl = d.ctl;
      Batch* store = d.sc.batch;
      int rst = reset;
      void* args[] = {&ctl, &bt, &store, &rst};
      cudaKernelNodeParams kp;
      memset(&kp, 0, sizeof(kp));
      kp.func = (void*)k_begin;
      kp.gridDim = dim3(1);
      kp.blockDim = dim3(1);
      kp.kernelParams = args;
      if (cudaGraphExecKernelNodeSetParams(g.exec, g.begin, &kp) != cudaSuccess) return ALTO_ECUDA;
      if (pm) {
        // fresh events at the timed stage boundaries
        StageClock clk(h, s);
        std::vector<cudaEvent_t> ev(g.ev_node.size(), nullptr);
        for (size_t k = 0; k < ev.size(); ++k) {
          if (!g.ev_node[k]) continue;
          ev[k] = clk.take();
          if (ev[k] && cudaGraphExecEventRecordNodeSetEvent(g.exec, g.ev_node[k], ev[k]) != cudaSuccess)
            return ALTO_ECUDA;
        }
        h->ev_pending.push_back(ev);
        for (int i = 0; i < ALTO_NUM_STAGES; ++i) h->stage_launches[i] += g.stage_launches[i];
      }
      if (cudaGraphLaunch(g.exec, s) != cudaSuccess) return ALTO_ECUDA;
      h->launches += g.launches;
      return ALTO_OK;
    }
  }
  PushRec rec(h, s);
  const int64_t launches = launch_push<false>(h, s, bt, reset, &rec, (u32)h->cfg.max_batch_fragments);
  if (h->profiling) {
    h->ev_pending.push_back(rec.clk.ev);
    for (int i = 0; i < ALTO_NUM_STAGES; ++i) h->stage_launches[i] += rec.stage_l[i];
  }
  h->launches += launches;
  if (cudaGetLastError() != cudaSuccess) return ALTO_ECUDA;
  return ALTO_OK;
}

alto_status alto_agg_drain(alto_agg_t* h, void* stream, alto_drain* out) {
  if (h == nullptr || out == nullptr) return ALTO_EINVAL;
  cudaStream_t s = (cudaStream_t)stream;
  memset(out, 0, sizeof(*out));
  if (cudaMemcpyAsync(h->h_ctl, h->d.ctl, sizeof(Ctl), cudaMemcpyDeviceToHost, s) != cudaSuccess)
    return ALTO_ECUDA;
  if (cudaStreamSynchronize(s) != cudaSuccess) return ALTO_ECUDA;
  const Ctl& c = *h->h_ctl;
  out->first_batch = h->drain_first;
  out->n_batches = h->pushed - h->drain_first;
  h->drain_first = h->pushed;
  if (c.status != ALTO_OK) {
    h->latched = c.status;
    return c.status;
  }
  // the output counters are reset by the next push that launches work (its
  // first kernel); until then nothing new has been completed
  const bool fresh = !h->reset_pending;
  out->n_records = fresh ? (int64_t)c.rec_count : 0;
  out->records = h->d.out_rec;
  out->n_payload = fresh ? (int64_t)c.pay_count : 0;
  out->payload = h->d.out_pay;
  out->n_topk = fresh ? (int64_t)c.topk_count : 0;
  out->topk = h->d.out_topk;
  if (h->ring_rec[1] != nullptr) {
    // later pushes fill the other ring while the caller reads this one
    h->ring_cur ^= 1;
    h->d.out_rec = h->ring_rec[h->ring_cur];
    h->d.out_pay = h->ring_pay[h->ring_cur];
    h->d.out_topk = h->ring_topk[h->ring_cur];
  }
  h->reset_pending = true;
  return ALTO_OK;
}

alto_status alto_agg_stats(alto_agg_t* h, void* stream, int64_t* open_groups, int64_t* arena_used) {
  if (h == nullptr) return ALTO_EINVAL;
  cudaStream_t s = (cudaStream_t)stream;
  if (cudaMemcpyAsync(h->h_ctl, h->d.ctl, sizeof(Ctl), cudaMemcpyDeviceToHost, s) != cudaSuccess)
    return ALTO_ECUDA;
  if (cudaStreamSynchronize(s) != cudaSuccess) return ALTO_ECUDA;
  if (open_groups) *open_groups = (int64_t)h->h_ctl->live_groups;
  if (arena_used) *arena_used = (int64_t)h->h_ctl->arena_used;
  return h->h_ctl->status;
}

alto_status alto_agg_profile(alto_agg_t* h, int enable) {
  if (h == nullptr) return ALTO_EINVAL;
  if (enable) {
    if (h->last_stream || h->pushed) cudaStreamSynchronize(h->last_stream);
    collect_profile(h);
    h->profiling = true;
    h->profile_mode = (enable == ALTO_PROFILE_HOT) ? ALTO_PROFILE_HOT : ALTO_PROFILE_STAGES;
    h->prof_pushes = 0;
    h->launches = 0;
    for (int i = 0; i < ALTO_NUM_STAGES; ++i) {
      h->stage_ms[i] = 0.0;
      h->stage_launches[i] = 0;
    }
  } else {
    h->profiling = false;
  }
  return ALTO_OK;
}

alto_status alto_agg_profile_read(alto_agg_t* h, alto_profile* out) {
  if (h == nullptr || out == nullptr) return ALTO_EINVAL;
  if (cudaStreamSynchronize(h->last_stream) != cudaSuccess) return ALTO_ECUDA;
  collect_profile(h);
  out->pushes = h->prof_pushes;
  out->launches = h->launches;
  for (int i = 0; i < ALTO_NUM_STAGES; ++i) {
    out->stage_ms[i] = h->stage_ms[i];
    out->stage_launches[i] = h->stage_launches[i];
  }
  return ALTO_OK;
}

alto_status alto_agg_destroy(alto_agg_t* h) {
  if (h == nullptr) return ALTO_OK;
  cudaDeviceSynchronize();
  for (auto& ev : h->ev_pending)
    for (cudaEvent_t e : ev)
      if (e) cudaEventDestroy(e);
  for (cudaEvent_t e : h->ev_free) cudaEventDestroy(e);
  free_graphs(h);
  free_all(h, nullptr);
  cudaDeviceSynchronize();
  delete h;
  return ALTO_OK;
}

}  // extern "C"

// ===========================================================================
// One-shot aggregation without device allocation.
//
// For callers that may not allocate device memory at all: code that runs
// under a strict memory budget owned by another allocator (a serving process
// whose framework reserved all free memory up front), code on a real-time path
// where cudaMalloc's implicit synchronisation is not acceptable, or plug-ins
// that a host application loads without giving them an allocator.  They get
// one entry point that aggregates one self-contained batch (fresh state;
// groups that do not complete inside the batch are dropped) and writes the
// records straight into buffers the caller owns.  Every table, scratch array
// and arena chunk it needs lives in the static device array below, of fixed
// size; it calls no cudaMalloc/cudaFree.  The array is shared by every call in
// the process on a given device and keeps the previous call's contents, so
// each call clears what must start empty, and calls that overlap on the GPU
// (two streams at once) race on it.
// ===========================================================================
namespace {

constexpr u64 kNaBytes = 32ull << 20;        // size of the static scratch
constexpr u64 kNaMaxFragments = 4096;        // n per call
constexpr u64 kNaMaxGroupsLevels = 16384;    // n * depth per call
constexpr u64 kNaMaxPayload = 1ull << 18;    // n_payload per call
constexpr u64 kNaTableSlots = 1ull << 15;    // open-group table slots
constexpr u64 kNaArenaElems = 1ull << 20;    // arena int32 elements

}  // namespace

static __device__ __align__(256) unsigned char g_noalloc_scratch[kNaBytes];

namespace {

struct NaDevice {
  bool ready;
  unsigned char* base;  // device address of g_noalloc_scratch on that device
};
NaDevice g_na_dev[64];
std::mutex g_na_mu;  // first calls from several host threads set up one entry once

struct NaCarver {
  unsigned char* base;
  u64 used = 0;
  bool ok = true;
  template <class T>
  T* take(u64 count) {
    u64 bytes = ((sizeof(T) * count + 255) / 256) * 256;
    if (bytes == 0) bytes = 256;
    T* p = base ? (T*)(base + used) : nullptr;
    used += bytes;
    if (used > kNaBytes) ok = false;
    return p;
  }
};

struct NaState {
  Dev d;
  SortBuffers leaf_sort, up_sort;
  LookbackState lbs;
  u64 T, PS, done_cap, dense_cap, sort_tiles, scan_tiles;
  int tbits;
};

// Carve every buffer of the one-shot pipeline out of the static scratch (a
// null base only measures).
void na_layout(const alto_agg_config& cfg, unsigned char* base, NaState& st, NaCarver& cv) {
  cv.base = base;
  const int D = cfg.depth;
  int concat = -1, kk = 0;
  bool has_score = false;
  for (int l = 0; l < D; ++l) {
    if (cfg.payload_op[l] == ALTO_PAYLOAD_CONCAT) concat = l;
    if (cfg.score_op[l] != ALTO_SCORE_NONE) has_score = true;
    if (cfg.score_op[l] == ALTO_SCORE_TOPK) kk = std::max(kk, (int)cfg.topk_k[l]);
  }
  const u64 nmax = kNaMaxFragments, T = kNaTableSlots;
  st.T = T;
  st.tbits = ilog2(T);
  st.done_cap = nmax * (u64)D;
  st.dense_cap = kNaMaxGroupsLevels;  // children of every level of one self-contained batch
  st.PS = next_pow2(std::max<u64>(2 * nmax * (u64)D, 1024));
  st.sort_tiles = nmax / 4096 + 2;
  st.scan_tiles = std::max<u64>(std::max<u64>(st.done_cap, st.dense_cap), nmax) / kScanTile + 2;
  Dev& d = st.d;
  memset(&d, 0, sizeof(d));
  d.ctl = cv.take<Ctl>(1);
  d.tab.key = cv.take<u64>(T);
  d.tab.hot = cv.take<Hot>(T);
  d.tab.done_idx = cv.take<u32>(T);
  if (concat >= 0) {
    d.tab.vec_n = cv.take<u32>(2 * T);
    d.tab.dir = cv.take<u32>(T * kVecs * kNumChunks);
  }
  if (kk > 0) d.tab.topk = cv.take<u64>(T * (u64)kk);
  d.tab.chain_len = std::max((D - 1 + 1) & ~1, 2);  // even: read as 16-byte pairs
  d.tab.chain = cv.take<u64>(T * (u64)d.tab.chain_len);
  d.tab.cbits = cv.take<u64>(4 * T);
  d.tab.cur = cv.take<u64>(T);
  d.tab.dbase = cv.take<u64>(T);
  d.tab.bstate = cv.take<uint4>(T);
  d.tab.ready = cv.take<u32>(T);
  d.tab.leaf_level = D - 1;
  d.tab.mask = (u32)(T - 1);
  d.tab.kk = kk;
  d.tab.max_probe = (int)T;
  if (concat >= 0) {
    d.ar.elems = kNaArenaElems;
    d.ar.pool = cv.take<int32_t>(kNaArenaElems);
    u64 off = 0;
    for (int j = 0; j < kNumChunks; ++j) {
      d.ar.stack_off[j] = off;
      d.ar.stack_cap[j] = kNaArenaElems / (1ull << (kChunk0Log + j)) + 1;
      off += d.ar.stack_cap[j];
    }
    d.ar.stack = cv.take<u32>(off);
  }
  d.cfg.depth = D;
  d.cfg.concat_level = concat;
  for (int l = 0; l < kMaxDepth; ++l) {
    d.cfg.score_op[l] = (l < D) ? cfg.score_op[l] : 0;
    d.cfg.topk_k[l] = (l < D && cfg.score_op[l] == ALTO_SCORE_TOPK) ? cfg.topk_k[l] : 0;
  }
  d.cfg.has_score = has_score;
  d.cfg.n_max = (u32)nmax;
  d.cfg.dense_cap = st.dense_cap;
  d.cfg.spin_limit = cfg.spin_limit > 0 ? (u64)cfg.spin_limit : (1ull << 20);
  Scratch& sc = d.sc;
  for (int b = 0; b < 2; ++b) {
    st.leaf_sort.keys[b] = cv.take<u32>(nmax);
    st.leaf_sort.vals[b] = cv.take<u32>(nmax);
    st.up_sort.keys[b] = cv.take<u32>(nmax);
    st.up_sort.vals[b] = cv.take<u32>(nmax);
  }
  st.leaf_sort.hist = cv.take<u32>(4 * 256);
  st.leaf_sort.bin_base = cv.take<u32>(4 * 256);
  st.leaf_sort.lookback = cv.take<u64>(st.sort_tiles * 256);
  st.leaf_sort.lb_tiles = st.sort_tiles;
  st.up_sort.hist = st.leaf_sort.hist;
  st.up_sort.bin_base = st.leaf_sort.bin_base;
  st.up_sort.lookback = st.leaf_sort.lookback;
  st.up_sort.lb_tiles = st.sort_tiles;
  sc.leaf_sort_keys0 = st.leaf_sort.keys[0];
  sc.up_sort_keys0 = st.up_sort.keys[0];
  sc.leaf_seg_start = cv.take<u32>(nmax + 1);
  sc.leaf_seg_of = cv.take<u32>(nmax);
  sc.up_seg_start = cv.take<u32>(nmax + 1);
  sc.up_list2 = cv.take<u32>(nmax);
  for (int b = 0; b < 2; ++b) {
    sc.it_rep[b] = cv.take<u32>(nmax);
    sc.it_cseq[b] = cv.take<u32>(nmax);
    sc.it_skey[b] = cv.take<u32>(nmax);
  }
  sc.seg_vb0 = cv.take<u32>(nmax);
  sc.seg_vb1 = cv.take<u32>(nmax);
  sc.seg_carry = cv.take<u32>(nmax);
  sc.leaf_pos = cv.take<u32>(nmax);
  sc.mask = cv.take<u32>((nmax + 31) / 32 * 32);
  sc.mblk = cv.take<u32>(nmax / 32 + 1);
  sc.prefix = cv.take<u32>(nmax);
  const u64 dc = st.done_cap;
  sc.done_e = cv.take<u32>(dc);
  sc.done_lvl = cv.take<u32>(dc);
  sc.done_cseq = cv.take<u32>(dc);
  sc.done_rank = cv.take<u32>(dc);
  sc.r_done = cv.take<u32>(dc);
  sc.r_dense_n = cv.take<u32>(dc);
  sc.r_topk_n = cv.take<u32>(dc);
  sc.r_meta_n = cv.take<u32>(dc);
  sc.r_dense_base = cv.take<u64>(dc + 1);
  sc.r_topk_off = cv.take<u64>(dc + 1);
  sc.r_arena_base = cv.take<u64>(dc + 1);
  if (concat >= 0) {
    sc.dense = cv.take<uint4>(st.dense_cap);
    sc.dst = cv.take<u64>(st.dense_cap + 1);
  }
  if (concat >= 0 && concat < D - 1) {
    sc.c_dense_base = cv.take<u64>(dc + 1);
    sc.c_arena_base = cv.take<u64>(dc + 1);
    d.tab.par = cv.take<u32>(T);
    d.tab.cidx = cv.take<u32>(T);
    d.tab.app = cv.take<u64>(T);
  }
  sc.pairset = cv.take<u64>(st.PS);
  sc.ps_mask = st.PS - 1;
  sc.done_cap = (u32)dc;
  // a one-shot batch is never longer than a warp's segment share
  sc.big_cap = (u32)(nmax / kBigSeg + 1);
  sc.big_seg = cv.take<u32>((u64)D * sc.big_cap);
  st.lbs.desc = cv.take<ulonglong2>(3 * st.scan_tiles);
  st.lbs.tiles = st.scan_tiles;
}

// Clear, in one launch, what every call must find empty: the control block
// (keeping its epoch), the table keys, the per-batch accumulators, the
// completion masks, the leaf-slot set, the free-chunk stacks and the sort
// histogram.  The arrays that are read by epoch stamp (the dense child slots
// and the per-entry placement state) are cleared too: where they sit in the
// static array depends on the depth, the CONCAT level and k, so after a call
// with another layout they would hold whatever that call left there, and a
// leftover token or key equal to the coming epoch would read as a stamp.
__global__ void k_na_reset(Dev d, u32* hist, u64 T, u64 PS, u32 nmax) {
  pdl_enter();
  const u64 tid = (u64)blockIdx.x * blockDim.x + threadIdx.x;
  const u64 stride = (u64)gridDim.x * blockDim.x;
  if (tid == 0) {
    Ctl* c = d.ctl;
    const u32 ep = c->epoch;
    unsigned char* p = (unsigned char*)c;
    for (size_t i = 0; i < sizeof(Ctl); ++i) p[i] = 0;
    c->epoch = ep;
  }
  for (u64 i = tid; i < T; i += stride) {
    d.tab.key[i] = kEmpty;
    uint4* hw = reinterpret_cast<uint4*>(d.tab.hot + i);
    hw[0] = make_uint4(0, 0, kNone, 0);
    hw[1] = make_uint4(0, 0, 0, 0);
    hw[2] = make_uint4(kNone, 0, 0, 0);
    hw[3] = make_uint4(0, 0, 0, 0);
    d.tab.cur[i] = 0;
    d.tab.ready[i] = 0;
  }
  for (u64 i = tid; i < PS; i += stride) d.sc.pairset[i] = 0;
  for (u64 i = tid; i < (nmax + 31) / 32 * 32; i += stride) d.sc.mask[i] = 0;
  for (u64 i = tid; i < nmax / 32 + 1; i += stride) d.sc.mblk[i] = 0;
  for (u64 i = tid; i < 4 * 256; i += stride) hist[i] = 0;
  for (u64 i = tid; i < T; i += stride) d.tab.bstate[i] = make_uint4(0, 0, 0, 0);
  if (d.sc.dense != nullptr)
    for (u64 i = tid; i < d.cfg.dense_cap; i += stride) d.sc.dense[i] = make_uint4(0, 0, 0, 0);
}

// Counts of the call for the caller: {status, records, payload, top-k pairs}.
__global__ void k_na_finish(const Ctl* ctl, int64_t* out) {
  pdl_enter();
  out[0] = ctl->status;
  out[1] = (ctl->status == ALTO_OK) ? (int64_t)ctl->rec_count : 0;
  out[2] = (ctl->status == ALTO_OK) ? (int64_t)ctl->pay_count : 0;
  out[3] = (ctl->status == ALTO_OK) ? (int64_t)ctl->topk_count : 0;
}

}  // namespace

extern "C" alto_status alto_agg_oneshot_noalloc(const alto_agg_config* cfg_in, const alto_batch* b,
                                                 alto_record* out_records, int64_t cap_records,
                                                 int32_t* out_payload, int64_t cap_payload,
                                                 alto_topk_pair* out_topk, int64_t cap_topk,
                                                 int64_t* out_counts, void* stream) {
  if (cfg_in == nullptr || b == nullptr || out_counts == nullptr) return ALTO_EINVAL;
  alto_agg_config cfg = *cfg_in;
  if (cfg.max_batch_fragments == 0) cfg.max_batch_fragments = (int64_t)kNaMaxFragments;
  if (cfg.max_batch_payload == 0) cfg.max_batch_payload = (int64_t)kNaMaxPayload;
  if (cfg.flags != 0) return ALTO_EINVAL;  // one batch: nothing to release in a stream
  alto_status v = validate(&cfg);
  if (v != ALTO_OK) return v;
  if (b->depth != cfg.depth || b->n < 0 || b->n_payload < 0) return ALTO_EINVAL;
  if (cap_records < 0 || cap_payload < 0 || cap_topk < 0) return ALTO_EINVAL;
  if ((cap_records > 0 && !out_records) || (cap_payload > 0 && !out_payload) ||
      (cap_topk > 0 && !out_topk))
    return ALTO_EINVAL;
  // sizes beyond what the static scratch holds
  if ((u64)b->n > kNaMaxFragments || (u64)b->n * (u64)cfg.depth > kNaMaxGroupsLevels ||
      (u64)b->n_payload > kNaMaxPayload)
    return ALTO_ENOSPC;
  if (b->n > 0 && (b->tags == nullptr || b->payload_off == nullptr)) return ALTO_EINVAL;
  if (b->n_payload > 0 && b->payload == nullptr) return ALTO_EINVAL;
  bool has_score = false;
  for (int l = 0; l < cfg.depth; ++l) has_score |= cfg.score_op[l] != ALTO_SCORE_NONE;
  if (b->n > 0 && has_score && b->score == nullptr) return ALTO_EINVAL;

  // once per device, with that device current: the static array's address
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return ALTO_ECUDA;
  unsigned char* base = nullptr;
  {
    std::lock_guard<std::mutex> lock(g_na_mu);
    NaDevice& nd = g_na_dev[dev];
    if (!nd.ready) {
      void* ptr = nullptr;
      if (cudaGetSymbolAddress(&ptr, g_noalloc_scratch) != cudaSuccess || ptr == nullptr)
        return ALTO_ECUDA;
      if (sort_prepare() != cudaSuccess) return ALTO_ECUDA;
      nd.base = (unsigned char*)ptr;
      nd.ready = true;
    }
    base = nd.base;
  }
  int num_sms = 0;
  if (cudaDeviceGetAttribute(&num_sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
    return ALTO_ECUDA;

  NaState st;
  NaCarver cv;
  na_layout(cfg, base, st, cv);
  if (!cv.ok) return ALTO_ENOSPC;
  Dev d = st.d;
  d.out_rec = out_records;
  d.out_pay = out_payload;
  d.out_topk = out_topk;
  d.cfg.out_records = (u64)cap_records;
  d.cfg.out_payload = (u64)cap_payload;
  d.cfg.out_topk = (u64)cap_topk;

  cudaStream_t s = (cudaStream_t)stream;
  const u32 n = (u32)b->n;
  const u32 nmax = (u32)kNaMaxFragments;
  Batch bt;
  bt.tags = b->tags;
  bt.off = b->payload_off;
  bt.pay = b->payload;
  bt.score = d.cfg.has_score ? b->score : nullptr;
  bt.n = n;
  bt.n_payload = (u64)b->n_payload;

  launch_pdl(k_na_reset, num_sms * 2, kThreads, 0, s, d, st.leaf_sort.hist, st.T, st.PS, nmax);
  launch_pdl(k_begin, 1, 1, 0, s, d.ctl, bt, (Batch*)nullptr, 0);
  if (n > 0) {
    Pipeline p;
    p.d = d;
    p.leaf_sort = &st.leaf_sort;
    p.up_sort = &st.up_sort;
    p.lbs = st.lbs;
    p.num_sms = num_sms;
    p.nb = nmax;
    p.tbits = st.tbits;
    p.nmax = nmax;
    p.s = s;
    enqueue_batch<false>(p, bt);  // its last kernel also ends the batch
  } else {
    launch_pdl(k_end, 1, 1, 0, s, d.ctl);
  }
  launch_pdl(k_na_finish, 1, 1, 0, s, d.ctl, out_counts);
  if (cudaGetLastError() != cudaSuccess) return ALTO_ECUDA;
  return ALTO_OK;
}
