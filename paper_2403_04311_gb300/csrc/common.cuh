// Shared device definitions of the alto_agg CUDA library (sm_103a).
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "alto_agg.h"

namespace alto {

typedef uint32_t u32;
typedef uint64_t u64;

constexpr int kMaxDepth = ALTO_MAX_DEPTH;
constexpr int kMaxTopk = ALTO_MAX_TOPK;
constexpr u64 kEmpty = ~0ull;          // free hash slot
constexpr u64 kTomb = ~0ull - 1;       // deleted hash slot
constexpr u32 kNone = 0xFFFFFFFFu;     // no last child yet / invalid chunk
constexpr int kChunk0Log = 5;          // smallest arena chunk: 32 int32
constexpr int kNumChunks = 22;         // chunk classes 32 << 0 .. 32 << 21
constexpr int kVecs = 2;               // per CONCAT group: 0 = leaf meta, 1 = payload
constexpr int kSites = 64;             // launch sites sharing look-back state per batch
constexpr int kWarps = 8;              // warps per 256-thread block

// ---------------------------------------------------------------------------
// device control block (one per handle, device memory)
// ---------------------------------------------------------------------------
struct Ctl {
  // persistent across batches
  u64 seq_base;            // arrival index of the next batch's first fragment
  u64 rec_count;           // records in the output ring since the last drain
  u64 pay_count;           // payload elements in the ring since the last drain
  u64 topk_count;          // top-k pairs in the ring since the last drain
  u64 bump;                // arena elements handed out by the bump allocator
  u64 live_groups;         // open groups in the table
  u64 arena_used;          // arena elements held by open groups' chunks
  u32 epoch;               // batch counter, starts at 1
  int status;              // latched alto_status
  int batch_err;           // priority-encoded error of the current batch
  int abort;               // a device wait gave up: the rest of the batch is skipped
  int test_stall;          // ALTO_FLAG_TEST_STALL: look-back waits never see a predecessor
  int top[kNumChunks];     // free-chunk stack heights per class
  u32 tile_ctr[kSites];    // dynamic tile counters per launch site
  u32 exit_ctr[kSites];    // CTAs finished per launch site (resets tile_ctr)
  u32 last_ctr;            // CTAs finished in a multi-scan launch with a last-CTA step
  // per batch (device-computed sizes that later kernels read)
  u32 n;                   // fragments in the batch
  u32 n_items[kMaxDepth];  // items entering level l
  u32 n_segs[kMaxDepth];   // distinct level-l groups in the batch
  u32 n_done;              // groups completed by the batch
  u32 skip_dense;          // set when a capacity check failed for this batch
  u32 skip_rec;            // the record scans' capacity check failed: no records (with a
                           // split placement that check leaves skip_dense to the placement's own)
  int pre_err;             // split placement: batch_err as the leaf finalize left it
  u32 n_done_leaf;         // split placement: leaf parents completed (done list 0..n-1)
  u64 leaf_dense_total;    // split placement: its own totals (the record scans beside it
  u64 leaf_arena_total;    // write dense_total and arena_total, which it never reads)
  u32 fin_ctr;             // split placement: leaf finalize CTAs finished
  u32 last_ctr2;           // as last_ctr, for the split placement's scans
  u64 dense_total;         // children of CONCAT groups completing in this batch
  u64 arena_total;         // buffered leaves of those groups
  u64 pay_total;           // payload elements emitted by this batch
  u64 topk_total;          // top-k pairs emitted by this batch
  u64 n_emit;              // records ranked by this batch
  u64 chain_total;         // dense child slots of completing groups at levels M < l
  u64 chain_arena;         // their buffered child spans
  u64 bm_used;             // streaming release: words of the presence bitmaps handed out
  u32 n_big[kMaxDepth];    // segments of level l longer than a warp's share, for the block reduce
  u32 n_rel;               // streaming: small leaf segments left to the warp reduce
  u64 scan_total[kSites];  // totals written by scans
  u64 pay_base;            // pay_count when the batch started (the gather's base: the
                           // batch's end may move pay_count while the gather still runs)
};

// Programmatic dependent launch.  Every kernel of the library is launched
// with programmatic stream serialization and first waits here until its
// predecessor in the stream has completed and its memory is visible; nothing
// of a batch reads state before the wait.  No kernel triggers its successor
// early: the implicit trigger at exit already hides most of the boundary
// (launch and memory flush), and an early trigger lets the kernel after next
// take SM slots while two grids still run, which split one-wave grids into a
// ragged second wave.
__device__ __forceinline__ void pdl_enter() { asm volatile("griddepcontrol.wait;" ::: "memory"); }

// error priority: the class reported when a batch holds several defects
__device__ __forceinline__ int err_priority(int code) {
  switch (code) {
    case ALTO_EINVAL: return 10;
    case ALTO_EDUP: return 9;
    case ALTO_EINCONSIST: return 8;
    case ALTO_ELAST: return 7;
    case ALTO_ECLOSED: return 6;
    case ALTO_ENOSPC: return 5;
    case ALTO_ETIMEOUT: return 4;
    default: return 1;
  }
}

__device__ __forceinline__ void raise_err(Ctl* ctl, int code) {
  atomicMax(&ctl->batch_err, (err_priority(code) << 8) | (-code));
}

// A wait that ran past its cap: record ETIMEOUT and stop the batch.
__device__ __forceinline__ void raise_timeout(Ctl* ctl) {
  raise_err(ctl, ALTO_ETIMEOUT);
  *(volatile int*)&ctl->abort = 1;
}

// Kernels of a batch do nothing once the handle is poisoned or a wait gave up.
__device__ __forceinline__ bool halted(const Ctl* c) {
  return c->status != ALTO_OK || *(const volatile int*)&c->abort != 0;
}

// IEEE-754 totalOrder key of a non-NaN float: larger key = larger value,
// -0.0 below +0.0.
__device__ __forceinline__ u32 score_key(float x) {
  u32 u = __float_as_uint(x);
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}
__device__ __forceinline__ float key_score(u32 k) {
  return __uint_as_float((k & 0x80000000u) ? (k & 0x7FFFFFFFu) : ~k);
}
__device__ __forceinline__ bool is_nan_bits(u32 u) { return (u & 0x7FFFFFFFu) > 0x7F800000u; }

// tag fields
__device__ __forceinline__ u32 tag_pid(u64 t) { return (u32)(t >> 32); }
__device__ __forceinline__ u32 tag_child(u64 t) { return (u32)t & 0x7FFFFFFFu; }
__device__ __forceinline__ u32 tag_last(u64 t) { return ((u32)t >> 31) & 1u; }

// splitmix64 finalizer (Steele, Lea, Flood 2014)
__device__ __forceinline__ u64 mix64(u64 x) {
  x ^= x >> 30;
  x *= 0xbf58476d1ce4e5b9ull;
  x ^= x >> 27;
  x *= 0x94d049bb133111ebull;
  x ^= x >> 31;
  return x;
}

__device__ __forceinline__ u32 lanemask_lt() {
  u32 m;
  asm("mov.u32 %0, %%lanemask_lt;" : "=r"(m));
  return m;
}

// Arena geometry: vector position x lives in chunk j = floor(log2(x/32 + 1)),
// which starts at position 32 * (2^j - 1) and holds 32 << j elements.
__device__ __forceinline__ int chunk_of(u64 x) {
  u64 q = (x >> kChunk0Log) + 1;
  return 63 - __clzll((long long)q);
}
__device__ __forceinline__ u64 chunk_start(int j) { return ((1ull << j) - 1) << kChunk0Log; }
__device__ __forceinline__ u64 chunk_size(int j) { return 1ull << (kChunk0Log + j); }

// ---------------------------------------------------------------------------
// device-resident state, handed to kernels by value
// ---------------------------------------------------------------------------
// The fields of an open-group entry that the level kernels read and write
// together, in one 64-byte record (one access brings them all; a
// structure-of-arrays table spread them over a dozen cache lines).  The
// batch accumulators are zero between batches (acc_fmin: kNone), also in
// free slots, so an insert made while other threads may already add to the
// new entry (a publishing insert) leaves them, and `touch`, alone.
struct __align__(64) Hot {
  u64 up;          // tag one level up
  u32 last;        // last child index or kNone
  u32 completed;   // complete children so far
  u64 acc_cl;      // this batch: complete children << 40 | payload elements (leaf level)
  u32 acc_m1;      // this batch: largest child index + 1
  u32 acc_cs1;     // this batch: largest completion seq + 1 of complete children
  u32 acc_fmin;    // this batch: smallest flagged child index (kNone = none)
  u32 acc_fmax1;   // this batch: largest flagged child index + 1 (0 = none)
  u32 acc_smx;     // this batch: largest score key of complete children
  u32 acc_rep;     // this batch: a representative fragment
  u32 maxc1;       // largest child index seen + 1
  u32 smax;        // largest score key over complete children (0 = none)
  u32 touch;       // epoch of the batch that last touched the entry (upper levels)
  u32 done_epoch;  // epoch of the batch that completed the group
};
static_assert(sizeof(Hot) == 64, "one 64-byte record per entry");

struct Table {
  u64* key;        // [T] (level << 32 | parent_id), kEmpty, kTomb
  Hot* hot;        // [T]
  u32* done_idx;   // [T] index in the batch's done list
  u32* vec_n;      // [T][2] CONCAT level: leaves in meta vector, elements in payload vector
  u32* dir;        // [T][2][kNumChunks] CONCAT level: chunk offsets in the arena
  u64* topk;       // [T][kk] TOPK levels: best (score_key << 32 | ~child) first
  u64* chain;      // [T][D-1] tags 0..l-1 of the group's first fragment (ancestry)
  u64* cur;        // [T] arena cursor: leaves << 40 | payload elements
  u64* dbase;      // [T] first dense child slot of a group completing this batch
  uint4* bstate;   // [T] where this batch's leaves go, one load per fragment:
                   //     {epoch, mode (1 arena, 2 dense), dense base lo, hi}
  // CONCAT at a level M above the leaf parent: a group of a level l with
  // M < l <= D-1 that completes is appended, as one child span, to its
  // parent's arena vectors (the parent's cursor `cur` counts the spans)
  u32* par;        // [T] parent entry the completed group was appended to
  u32* cidx;       // [T] its child index in that parent
  u64* app;        // [T] its reserved place there: span index << 40 | payload position
  // [T][4] leaf parents: leaf slots 0..255 seen while the group is open (kept
  // apart from the chain rows: sharing their lines with these atomics made the
  // leaf accumulate slower)
  u64* cbits;
  // streaming release (CONCAT at the leaf parent): children 0..rel-1 were
  // released by partial records and are no longer buffered; rnew is where
  // the release of the current batch ends (a partial or the final record)
  u32* rel;        // [T]
  u32* rnew;       // [T]
  // [T] 1 once a publishing insert has written the entry's chain row (0
  // while the slot is free): a finder in the launch that inserts the entry
  // compares ancestry only after that
  u32* ready;
  int leaf_level;  // D - 1
  int chain_len;   // D - 1, rounded up to even
  u32 mask;        // T - 1
  int kk;          // stride of topk (largest k over levels)
  int max_probe;
};

struct Arena {
  int32_t* pool;        // [A]
  u32* stack;           // concatenated per-class free stacks
  u64 stack_off[kNumChunks];
  u64 stack_cap[kNumChunks];
  u64 elems;            // A
};

struct Cfg {
  int depth;
  int concat_level;     // -1 if none
  int score_op[kMaxDepth];
  int topk_k[kMaxDepth];
  bool has_score;
  bool stream;          // streaming release at the CONCAT level
  bool stream_leaf;     // ... and that level is the leaf parent (the sorted leaf path releases)
  u32 n_max;
  u64 out_records, out_payload, out_topk, dense_cap;
  u64 spin_limit;
};

}  // namespace alto
