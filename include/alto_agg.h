/*
 * alto_agg -- batched re-aggregation of streamed fragments by nested ancestry
 * on one GPU (NVIDIA GB300, sm_103a).
 *
 * The operation follows Alto (arxiv 2403.04311):
 *   - Sec. 4.2: every parallel-map (pmap) entry pushes one ancestry tag on
 *     each element -- the id of the parent element and the element's index in
 *     the parent's stream -- and every pmap exit pops one tag and aggregates
 *     the outputs of that call.  A fragment therefore carries D tags, one per
 *     nesting level, outermost first.
 *   - Sec. 3.1: a stream is known to be complete only when its end-of-output
 *     delimiter arrives.  Here the delimiter is the last-flag bit on the tag of
 *     the stream's final child.
 *   - Sec. 3.2 / Sec. 4.1: the outputs of a pmap are reconstituted in the
 *     original stream order.  Sec. 3.3: an aggregate operator collects one
 *     stream's items into one output object.  Sec. 4.3: all elements with the
 *     same ancestry are routed to the same aggregation point.
 *
 * Data model.  Tag l of a fragment is packed into a u64 as
 *     parent_id << 32 | last << 31 | child_index        (child_index < 2^31)
 * The fragment is child `child_index` of group (l, parent_id).  For l < D-1
 * that child is the group (l+1, parent_id of tag l+1); for l = D-1 the child
 * is the fragment itself (a leaf, complete on arrival).  parent_ids are unique
 * per level over the aggregator's lifetime, and a group always sits under the
 * same tag one level up.  A group is complete when some child carries the
 * last flag (index `last`), every child 0..last is present, and every child is
 * complete.  Completed groups are emitted, at every level, as one record each:
 *   - CONCAT (at most one level M): the payloads of the subtree's leaves
 *     concatenated in child-index path order;
 *   - MAX: the record's score is the largest leaf score of the subtree;
 *   - TOPK(k): also the k children with the largest score (a child's score is
 *     the largest leaf score of its subtree), ties to the smaller child index.
 * Scores are compared under IEEE-754 totalOrder (-0.0 < +0.0); NaN is
 * rejected.  Groups with no operation still emit a record (empty payload).
 *
 * Emission order.  Within a push, records come in (completion_seq ascending,
 * level descending) order, where completion_seq is the global arrival index of
 * the fragment that completed the group (the largest arrival index in its
 * subtree).  Records of successive pushes follow one another.  Batches are
 * taken in push order; fragments of a batch in array order.
 *
 * Streams.  Every call takes a CUDA stream (a cudaStream_t passed as void*).
 * push_batch only enqueues work; drain is the only call that synchronises.
 * Device buffers passed to push_batch are borrowed until the work enqueued on
 * that stream has completed, exactly like cudaMemcpyAsync.  A handle is not
 * thread-safe.
 *
 * Errors.  Every call returns an alto_status.  Argument errors found on the
 * host are returned at once and leave the handle usable.  Errors found on the
 * device are latched: the first batch with an error poisons the handle, the
 * next drain returns the error (with no records), and every later call
 * returns it too; destroy still succeeds.  When one batch holds several
 * defects the reported class is the first of EINVAL, EDUP, EINCONSIST, ELAST,
 * ENOSPC, ETIMEOUT.  Device detection covers: offsets that decrease or end
 * beyond n_payload, NaN scores (EINVAL); a leaf (group, child index) given
 * twice in one batch, and -- for CONCAT groups -- a repeated or missing child
 * found when the group completes (EDUP); a group seen under two different
 * parent tags, or two different child groups in one slot within one batch
 * (EINCONSIST); two different last children, or a child index above the last
 * (ELAST); table, arena or output capacity exceeded (ENOSPC); a device-side
 * wait that ran past its iteration cap (ETIMEOUT).  A full open-group table
 * and a wait that ran out stop the batch where they happen, so a defect that
 * would be found later in the same batch is not reported.  Inputs outside
 * that scope (for example a fragment for a group that was already emitted)
 * give undefined records but never a fault or a hang.
 */
#ifndef ALTO_AGG_H
#define ALTO_AGG_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef int alto_status;

#define ALTO_OK 0
#define ALTO_EINVAL (-1)     /* bad argument, offsets or NaN score */
#define ALTO_ENOMEM (-2)     /* device allocation failed */
#define ALTO_ENOSPC (-3)     /* table, arena or output capacity exceeded */
#define ALTO_EDUP (-4)       /* the same leaf slot given twice */
#define ALTO_ELAST (-5)      /* conflicting last child, or a child past it */
#define ALTO_EINCONSIST (-6) /* a group under two parent tags / a slot with two children */
#define ALTO_ECLOSED (-7)    /* fragment for an emitted group (not detected on the device) */
#define ALTO_ETIMEOUT (-8)   /* a device-side wait hit its iteration cap */
#define ALTO_ECUDA (-9)      /* a CUDA runtime call failed */

#define ALTO_MAX_DEPTH 8
#define ALTO_MAX_TOPK 32

#define ALTO_PAYLOAD_NONE 0
#define ALTO_PAYLOAD_CONCAT 1
#define ALTO_SCORE_NONE 0
#define ALTO_SCORE_MAX 1
#define ALTO_SCORE_TOPK 2

/* Streaming release (flags bit 0; Sec. 3.2: the outputs of a pmap are put
 * back in order and passed on as a stream).  Every push also emits, for each
 * still-open group of the CONCAT level whose run of complete children
 * 0..r-1 grew past the r it released before, a partial record: ops = CONCAT
 * | ALTO_OPS_PARTIAL, n_children = r, payload = the newly released children's
 * concatenations in child order, score 0, no top-k, completion_seq = the
 * latest completion seq among those children (at the leaf parent, the latest
 * arrival).  The group's final record then carries only the children not
 * released before (its other fields are unchanged).  Records stay in
 * (completion_seq, deeper first) order.  EINVAL with no CONCAT level and for
 * alto_agg_oneshot_noalloc. */
#define ALTO_FLAG_STREAM_RELEASE 1
#define ALTO_OPS_PARTIAL 0x80

/* Two output rings (flags bit 1): pushes fill one ring while the records,
 * payload and top-k pairs of the previous drain stay in the other, and every
 * drain swaps them.  What a drain returns then stays valid through the next
 * drain, until the first push after it (or destroy), instead of until the
 * next push, so the caller can copy it out while later pushes run.  Takes
 * twice the output capacities' memory.  EINVAL for alto_agg_oneshot_noalloc. */
#define ALTO_FLAG_DOUBLE_RING 2

/* Failure-path test hook (flags bit 2; the paper has no counterpart): every
 * look-back wait of a push (the scans' and the radix sort's) waits on a
 * predecessor's descriptor that nothing publishes, so the first wait of a
 * scan or sort with more than one tile polls spin_limit times, records
 * ALTO_ETIMEOUT and stops the batch, as a wait that really ran out does.  The
 * next drain returns ALTO_ETIMEOUT and the handle stays poisoned; destroy
 * still succeeds and the CUDA context stays usable.  Only for testing the
 * timeout path: leave it off.  EINVAL for alto_agg_oneshot_noalloc. */
#define ALTO_FLAG_TEST_STALL 4

/* Launch every kernel of a push one by one (flags bit 3).  By default a push
 * of at most 131,072 fragments replays a CUDA graph of its launch sequence,
 * captured on the handle's first such push (per output ring and profiling
 * mode): one host launch per push instead of about twenty.  Larger pushes
 * always launch directly.  Results are the same either way.  EINVAL for
 * alto_agg_oneshot_noalloc, which always launches directly. */
#define ALTO_FLAG_DIRECT_LAUNCH 8

/* Aggregator configuration (Sec. 5: the controller is told which queues are
 * pmap entry/exit points and which data is aggregated; here: the nesting
 * depth and what each level's exit computes).  Zero capacities take the
 * defaults noted. */
typedef struct alto_agg_config {
  int32_t depth;                          /* D, number of tags, 1..8 */
  int32_t payload_op[ALTO_MAX_DEPTH];     /* per level: NONE or CONCAT (at most one level) */
  int32_t score_op[ALTO_MAX_DEPTH];       /* per level: NONE, MAX or TOPK */
  int32_t topk_k[ALTO_MAX_DEPTH];         /* per TOPK level: 1..32 */
  int64_t max_batch_fragments;            /* largest n of one push (required, < 2^30) */
  int64_t max_batch_payload;              /* largest n_payload of one push (required) */
  int64_t max_open_groups;                /* groups alive at once (default 2^20) */
  int64_t arena_elems;                    /* int32 elements buffered for open CONCAT groups (default 2^26) */
  int64_t out_records;                    /* records held between drains (default 4*max_batch_fragments) */
  int64_t out_payload_elems;              /* payload elements held between drains (default 4*max_batch_payload) */
  int64_t out_topk;                       /* top-k pairs held between drains (default out_records) */
  int64_t max_emit_children;              /* children of CONCAT groups completing in one push (default 4*max_batch_fragments) */
  int64_t spin_limit;                     /* device wait cap in polls (default 2^20) */
  int64_t flags;                          /* ALTO_FLAG_* (0: none) */
} alto_agg_config;

/* Device memory provider.  alloc returns device memory of at least `bytes`
 * usable on `stream` (or NULL); free releases it.  A NULL allocator means
 * cudaMallocAsync / cudaFreeAsync on the given stream. */
typedef struct alto_allocator {
  void* ctx;
  void* (*alloc)(void* ctx, size_t bytes, void* stream);
  void (*free)(void* ctx, void* ptr, void* stream);
} alto_allocator;

/* One batch of fragments, all pointers to device memory.
 *   tags        [depth][n] u64, level-major: tag l of fragment i at tags[l*n + i]
 *   payload_off [n+1] u32 element offsets into payload; fragment i's payload is
 *               payload[payload_off[i] .. payload_off[i+1]); must not decrease,
 *               and payload_off[n] <= n_payload
 *   payload     [n_payload] int32 tokens
 *   score       [n] f32, required iff some level has a score op, else ignored */
typedef struct alto_batch {
  int64_t n;
  int32_t depth;
  int32_t reserved;
  const uint64_t* tags;
  const uint32_t* payload_off;
  int64_t n_payload;
  const int32_t* payload;
  const float* score;
} alto_batch;

/* One completed group (48 bytes).  payload_off / topk_off index the drain's
 * payload and top-k arrays.  score is the subtree's largest leaf score for
 * levels with a score op, else 0.  ops = payload_op | score_op << 2. */
typedef struct alto_record {
  uint64_t completion_seq;
  uint64_t payload_off;
  uint64_t payload_len;
  uint64_t topk_off;
  uint32_t parent_id;
  uint32_t n_children;
  uint8_t level;
  uint8_t ops;
  uint16_t topk_n;
  float score;
} alto_record;

/* A selected child: best score first, ties to the smaller child index. */
typedef struct alto_topk_pair {
  uint32_t child_index;
  float score;
} alto_topk_pair;

/* Everything completed since the previous drain.  All pointers are device
 * memory owned by the handle, valid until the next push, drain or destroy
 * (with ALTO_FLAG_DOUBLE_RING: through the next drain, until the first push
 * after it, or destroy). */
typedef struct alto_drain {
  int64_t n_records;
  const alto_record* records;
  int64_t n_payload;
  const int32_t* payload;
  int64_t n_topk;
  const alto_topk_pair* topk;
  uint64_t first_batch;   /* index of the first batch pushed since the previous drain */
  uint64_t n_batches;     /* batches pushed since the previous drain */
} alto_drain;

typedef struct alto_agg alto_agg_t;

/* Sec. 5 (the controller handles pmap tracking): allocate the open-group
 * table, the arena, scratch and the output ring for `cfg` through `alloc`
 * (NULL: cudaMallocAsync on `stream`), and return the handle in *out.
 * Errors: EINVAL (bad config; *out untouched), ENOMEM, ECUDA. */
alto_status alto_agg_create(const alto_agg_config* cfg, const alto_allocator* alloc,
                            void* stream, alto_agg_t** out);

/* Sec. 4.2-4.3: route the batch's fragments to their groups by ancestry,
 * merge them with the groups left open by earlier batches, decide completion
 * level by level, and append the records of every group completed by this
 * batch to the handle's output ring (Sec. 3.3).  Enqueues on `stream`, never
 * synchronises.  n = 0 is a no-op batch.  Host-side errors (returned at once,
 * handle still usable): EINVAL for a NULL handle or batch, depth mismatch,
 * n < 0 or n > max_batch_fragments, n_payload outside 0..max_batch_payload,
 * NULL tags/offsets with n > 0, NULL payload with n_payload > 0, NULL score
 * when a score op is configured.  A latched device error is returned as is. */
alto_status alto_agg_push_batch(alto_agg_t* h, const alto_batch* b, void* stream);

/* Synchronise `stream` and return, in *out, every record completed since the
 * previous drain (Sec. 3.3 aggregate output), in emission order, with its
 * payload and top-k pairs.  Returns the latched status; after an error *out
 * holds no records. */
alto_status alto_agg_drain(alto_agg_t* h, void* stream, alto_drain* out);

/* Open groups and buffered arena elements right now (synchronises stream). */
alto_status alto_agg_stats(alto_agg_t* h, void* stream, int64_t* open_groups,
                           int64_t* arena_elems_used);

/* Measurement hooks.  The paper has no counterpart: they exist so that the
 * benchmark can time the pipeline's stages on the device while it runs.
 * With profiling on, every push records CUDA events at stage boundaries on
 * its stream; alto_agg_profile_read synchronises the handle's last push
 * stream and sums the elapsed times.  Stages, in push order:
 *   0 ingest (validate, table lookup)      1 leaf sort (TOPK leaf level)
 *   2 leaf accumulate (or segments+reduce) 3 leaf finalize
 *   4 upper levels                         5 emission order + offsets
 *   6 arena carry-over (TOPK leaf level)   7 dense child placement + length scan
 *   8 payload gather                       9 records, frees, table sweep
 * `launches` counts every kernel the pushes launched (also when profiling is
 * off).  enable = ALTO_PROFILE_STAGES (1) records an event at every stage
 * boundary; ALTO_PROFILE_HOT (2) records only the events around the two
 * heaviest kernels, the leaf accumulate (stage 2) and the payload gather
 * (stage 8), so that the other kernel boundaries run as without profiling;
 * either starts a fresh count.  0 stops recording events. */
#define ALTO_NUM_STAGES 10
#define ALTO_PROFILE_OFF 0
#define ALTO_PROFILE_STAGES 1
#define ALTO_PROFILE_HOT 2
typedef struct alto_profile {
  int64_t pushes;                          /* pushes since the last enable */
  int64_t launches;                        /* kernels those pushes launched */
  double stage_ms[ALTO_NUM_STAGES];        /* summed device time per stage */
  int64_t stage_launches[ALTO_NUM_STAGES]; /* kernels per stage, summed */
} alto_profile;

alto_status alto_agg_profile(alto_agg_t* h, int enable);
alto_status alto_agg_profile_read(alto_agg_t* h, alto_profile* out);

/* One-shot aggregation that allocates no device memory.  The paper has no
 * counterpart: this entry point serves callers that may not call cudaMalloc
 * -- a serving process whose framework has already reserved the device's free
 * memory for its own pool, a real-time path that cannot take cudaMalloc's
 * implicit device synchronisation, a plug-in loaded without an allocator.
 *
 * It aggregates ONE self-contained batch exactly as create + push_batch +
 * drain would on a fresh handle (groups not completed by the batch are
 * dropped), writing records, payload and top-k pairs into the caller's device
 * buffers, and {status, n_records, n_payload, n_topk} into the caller's device
 * int64[4] `out_counts`, all on `stream` (nothing is synchronised; status is
 * ALTO_ENOSPC there when an output capacity is too small).  Its tables,
 * scratch and arena live in one static device array of 32 MiB that every GPU
 * loading this library holds until the process exits.  Limits: n <= 4096,
 * n * depth <= 16384, n_payload <= 262144; larger batches return ALTO_ENOSPC
 * at once.  The first call on a device looks up that array's device address
 * (cudaGetSymbolAddress) with the device current; make that first call before
 * any stream capture.  All calls on a device share the array and each call
 * clears what must start empty, so calls that overlap on the GPU (for
 * example on two streams at once) race and give undefined results.  Returns
 * ALTO_EINVAL for bad arguments, ALTO_ECUDA if a launch fails. */
alto_status alto_agg_oneshot_noalloc(const alto_agg_config* cfg, const alto_batch* b,
                                     alto_record* out_records, int64_t cap_records,
                                     int32_t* out_payload, int64_t cap_payload,
                                     alto_topk_pair* out_topk, int64_t cap_topk,
                                     int64_t* out_counts, void* stream);

/* Sec. 3.1: a stream is complete only once its end-of-output delimiter has
 * arrived, so a group whose last child never came cannot be emitted.  Free
 * everything the handle owns; such open groups are discarded.  NULL is OK.
 * Always succeeds on a valid or poisoned handle. */
alto_status alto_agg_destroy(alto_agg_t* h);

/* ---- split_text: the fragmentation step before the aggregator ------------
 *
 * Sec. 3.1-3.2 (the split_text operator turns a text item of a Delimiter type
 * into a stream of smaller Delimiter items, one level of hierarchy below it)
 * and Sec. 4.2 (at a pmap entry every child keeps its parent's tags and gets
 * one new tag).  Each of n_src token streams is cut after every delimiter
 * token; piece k of stream s becomes a fragment whose tags are the stream's
 * depth_in tags followed by (src_id[s], k, last = final piece).  A delimiter
 * stays at the end of the piece it closes; a stream that ends with a
 * delimiter has no trailing empty piece; an empty stream has one empty piece.
 * The pieces tile the streams, so they need no copy: out_off indexes the
 * input `tokens`, and {out_tags, out_off, tokens} is directly a batch for
 * alto_agg_push_batch (depth depth_in + 1, n = n_frag) with the pieces in
 * stream order.
 *
 * All pointers are device memory except `a` itself.  tok_off must start at 0,
 * be non-decreasing and end at n_tokens.  out_tags is level-major with stride
 * n_frag (the number of pieces, which the call computes): the caller gives
 * capacity for cap_frag pieces, (depth_in + 1) * cap_frag tags and cap_frag + 1
 * offsets.  Stream-ordered on `stream`, no synchronisation: the outcome is
 * written to the device int64 out_counts[2] = {status, n_frag}, status
 * ALTO_EINVAL for bad offsets, ALTO_ENOSPC when n_frag > cap_frag (nothing else
 * is written then; n_frag is still the count needed).  `scratch` is device
 * memory of at least alto_split_scratch_bytes(n_src, n_tokens) bytes, 256-byte
 * aligned, owned by the caller; calls sharing a scratch must not overlap.
 * `tokens` is read fastest 16-byte aligned (four tokens a load).  The
 * return value is ALTO_EINVAL for bad host arguments (n_delims outside
 * 1..ALTO_MAX_DELIMS, depth_in outside 0..ALTO_MAX_DEPTH-1, null pointers,
 * too little scratch), ALTO_ECUDA if a launch fails, else ALTO_OK. */
#define ALTO_MAX_DELIMS 32
typedef struct alto_split_args {
  int64_t n_src;              /* streams */
  int64_t n_tokens;           /* tokens of all streams */
  int32_t depth_in;           /* tags each stream carries, 0..ALTO_MAX_DEPTH-1 */
  int32_t n_delims;           /* delimiter token ids, 1..ALTO_MAX_DELIMS */
  int32_t delims[ALTO_MAX_DELIMS];
  const uint64_t* src_tags;   /* [depth_in * n_src] level-major; may be NULL if depth_in == 0 */
  const uint32_t* src_id;     /* [n_src] the streams' ids at the new level */
  const uint32_t* tok_off;    /* [n_src + 1] */
  const int32_t* tokens;      /* [n_tokens] */
  int64_t cap_frag;
  uint64_t* out_tags;         /* [(depth_in + 1) * n_frag] */
  uint32_t* out_off;          /* [n_frag + 1] */
  int64_t* out_counts;        /* [2]: status, n_frag */
  void* scratch;
  int64_t scratch_bytes;
} alto_split_args;

int64_t alto_split_scratch_bytes(int64_t n_src, int64_t n_tokens);
alto_status alto_split_text(const alto_split_args* a, void* stream);

/* ---- routing by ancestry: the step in front of replicated aggregators ----
 *
 * Sec. 4.3: the aggregation at a pmap exit needs every element of a group at
 * the same instance of the next stage, so all elements with the same
 * ancestry tags go to the same instance (like ECMP, keyed on the tags), and a
 * new flow may be placed by load instead of by a hash; Sec. 5: the
 * controller picks replicas by these rules and by queue lengths.
 *
 * A flow is the group at the routing level L: fragments whose tags agree on
 * levels 0..L (parent ids are unique per level, so (L, p_L) names it).
 * ALTO_ROUTE_HASH places it at splitmix64(L << 32 | p_L) mod R.
 * ALTO_ROUTE_LEAST_LOADED keeps a placed flow on its replica and deals the
 * batch's new flows, in the order of their first fragment, round-robin over
 * the replicas ordered by load at the start of the batch (fewest first, ties
 * to the lower index), the load being the fragments routed to the replica so
 * far.  alto_router_release forgets the flows whose groups the aggregator
 * reported complete.  Each batch is partitioned stably: replica r's
 * sub-batch holds its fragments in arrival order and is itself a batch for
 * alto_agg_push_batch.
 *
 * Calls are stream-ordered and do not synchronise, except
 * alto_router_counts.  Device-detected errors (bad payload offsets: EINVAL;
 * flow table full: ENOSPC; a wait that ran out: ETIMEOUT) latch and poison
 * the handle; the next call returns them. */
#define ALTO_ROUTE_HASH 0
#define ALTO_ROUTE_LEAST_LOADED 1
#define ALTO_MAX_REPLICAS 1024

typedef struct alto_router_config {
  int32_t depth;               /* tags per fragment, 1..ALTO_MAX_DEPTH */
  int32_t level;               /* routing level L, 0..depth-1 */
  int32_t n_replicas;          /* R, 1..ALTO_MAX_REPLICAS */
  int32_t policy;              /* ALTO_ROUTE_HASH or ALTO_ROUTE_LEAST_LOADED */
  int64_t max_batch_fragments; /* n per batch, >= 1 */
  int64_t max_batch_payload;   /* payload elements per batch */
  int64_t max_flows;           /* LEAST_LOADED: flows placed at once (0: 2^20) */
  int32_t with_score;          /* batches carry scores (routed along) */
  int32_t reserved;
} alto_router_config;

typedef struct alto_router alto_router_t;

/* The last batch's routing, all in device memory owned by the handle, valid
 * until the next route or destroy.  Replica r's sub-batch: n_r =
 * frag_off[r+1] - frag_off[r] fragments; tags at tags + depth * frag_off[r]
 * (level-major with stride n_r); payload_off at payload_off + frag_off[r] + r
 * (n_r + 1 offsets from 0); payload at payload + pay_off[r]; scores at
 * score + frag_off[r]. */
typedef struct alto_routed {
  const uint32_t* replica;     /* [n] replica of each input fragment */
  const uint32_t* perm;        /* [n] input fragments grouped by replica, in arrival order */
  const int64_t* frag_off;     /* [R + 1] */
  const int64_t* pay_off;      /* [R + 1] */
  const uint64_t* tags;        /* [depth * n] */
  const uint32_t* payload_off; /* [n + R] */
  const int32_t* payload;      /* [n_payload] */
  const float* score;          /* [n] or NULL */
} alto_routed;

alto_status alto_router_create(const alto_router_config* cfg, const alto_allocator* alloc, void* stream,
                               alto_router_t** out);
/* Route one batch (device buffers, borrowed until the stream reaches the work). */
alto_status alto_router_route(alto_router_t* h, const alto_batch* b, void* stream, alto_routed* out);
/* Synchronise and copy the last batch's frag_off and pay_off (R + 1 each) to
 * host arrays; returns the latched status. */
alto_status alto_router_counts(alto_router_t* h, void* stream, int64_t* frag_off, int64_t* pay_off);
/* Forget the flows of the groups in `records` (device, as a drain returns
 * them) that sit at the routing level. */
alto_status alto_router_release(alto_router_t* h, const alto_record* records, int64_t n_records, void* stream);
/* Free everything; NULL is OK. */
alto_status alto_router_destroy(alto_router_t* h);

#ifdef __cplusplus
}
#endif

#endif /* ALTO_AGG_H */
