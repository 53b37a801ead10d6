"""Seeded generators for the five fragment-stream workloads (and small variants).

Every stream is a forest of nested-ancestry trees (paper Sec. 4.2): a group at
level l has children indexed 0..last; for l < D-1 a child is itself a group
one level down, for l = D-1 a child is a leaf fragment.  Each leaf carries one
tag per level, (parent_id u32, child_index u31, last-flag bit), packed into a
u64 as ``parent_id << 32 | last << 31 | child_index``.  Tags are stored
level-major, ``tags[l, i]`` for fragment i in arrival order.

Recipes (numpy PCG64, seeded):

* ``tiny``      D=2, one source -> queries with U{1..8} sentences, exactly 4,096
  leaves (last query truncated), payload U{1..32} tokens, child order shuffled
  within each parent, one batch.  seed 1.
* ``tiny64``    the literal 64 queries x U{1..8} sentences variant.  seed 6.
* ``factcheck`` D=4, source -> 1,024 responses -> U{2..10} claims -> 5
  documents -> U{3..20} sentences; payload U{8..40}; score N(0,1); global
  random interleave; 64K batches.  seed 2.
* ``throughput`` D=4, one source per root (c0=0, last), Zipf(1.2) fanout capped
  at 256 on levels 1-3, payload U{1..64}; leaves shuffled inside each root and
  W roots interleaved round-robin, W bisected so that ~20% of the leaf-parent
  groups span a batch boundary; 16M leaves in 1M batches.  seed 3.
* ``tokens``    D=2, one source -> 4,096 streams x 24,414 single-token leaves,
  round-robin with seeded jitter (key t*4096 + s + floor(4096 u), stable);
  8K batches.  seed 4.
* ``adversarial`` D=6, one source per root, fanout U{1..4} on levels 1-5, plus
  one hot leaf-parent with 1,048,576 leaves spread uniformly over the stream;
  every group's last-flagged child subtree arrives U{0..3} batches early;
  payload U{1..16}; score N(0,1); 64M leaves in 2M batches.  seed 5.

Every generator takes ``n_leaves`` and ``batch`` so that tests can draw a
scaled-down stream with the same structure.
"""
from __future__ import annotations

import heapq
import os
from concurrent.futures import ThreadPoolExecutor
from dataclasses import dataclass, field

import numpy as np

TOKEN_VOCAB = 50257

# payload ops / score ops (same integer codes as the C-ABI config)
NONE, CONCAT = 0, 1
S_NONE, S_MAX, S_TOPK = 0, 1, 2

CONFIG_NAMES = ("tiny", "tiny64", "factcheck", "throughput", "tokens", "adversarial", "tot")

_U32 = np.uint64(0xFFFFFFFF)


_CHUNK = 1 << 24


def _integers(rng, low, high, size, dtype=np.int32):
    """Uniform integers drawn in parallel chunks from child seed sequences of
    one seed drawn from ``rng`` (deterministic, independent of thread count)."""
    if size <= _CHUNK:
        return rng.integers(low, high, size=size, dtype=dtype)
    seed = int(rng.integers(0, 2**63))
    n_chunks = (size + _CHUNK - 1) // _CHUNK
    children = np.random.SeedSequence(seed).spawn(n_chunks)
    out = np.empty(size, dtype=dtype)

    def fill(k):
        a, b = k * _CHUNK, min(size, (k + 1) * _CHUNK)
        out[a:b] = np.random.default_rng(children[k]).integers(low, high, size=b - a, dtype=dtype)

    with ThreadPoolExecutor(max_workers=min(n_chunks, os.cpu_count() or 1)) as ex:
        list(ex.map(fill, range(n_chunks)))
    return out


def pack_tags(pid, child, last):
    """Pack (parent_id, child_index, last) arrays into u64 tags."""
    pid = np.asarray(pid, dtype=np.uint64)
    child = np.asarray(child, dtype=np.uint64)
    last = np.asarray(last, dtype=np.uint64)
    return (pid << np.uint64(32)) | (last << np.uint64(31)) | child


@dataclass
class Stream:
    name: str
    depth: int
    payload_op: tuple
    score_op: tuple
    topk_k: tuple
    tags: np.ndarray          # (D, N) uint64, arrival order
    off: np.ndarray           # (N+1,) int64 global CSR into payload
    payload: np.ndarray       # int32 tokens
    score: np.ndarray | None  # (N,) float32 or None
    batch_sizes: np.ndarray   # int64 per batch
    meta: dict = field(default_factory=dict)

    @property
    def n(self) -> int:
        return int(self.tags.shape[1])

    @property
    def n_batches(self) -> int:
        return len(self.batch_sizes)

    def batch_starts(self) -> np.ndarray:
        return np.concatenate([[0], np.cumsum(self.batch_sizes)]).astype(np.int64)

    def batch(self, b: int) -> dict:
        """Batch b as the C-ABI expects it: level-major tags (D*n), u32 CSR
        rebased to the batch's own payload slice, the payload slice, scores."""
        st = self.batch_starts()
        s, e = int(st[b]), int(st[b + 1])
        p0, p1 = int(self.off[s]), int(self.off[e])
        return dict(
            n=e - s,
            seq_base=s,
            tags=np.ascontiguousarray(self.tags[:, s:e]),
            off=(self.off[s:e + 1] - p0).astype(np.uint32),
            payload=self.payload[p0:p1],
            score=None if self.score is None else self.score[s:e],
        )

    def ops(self) -> dict:
        return dict(depth=self.depth, payload_op=list(self.payload_op),
                    score_op=list(self.score_op), topk_k=list(self.topk_k))


# ----------------------------------------------------------------------------
# tree construction
# ----------------------------------------------------------------------------

def _children(counts):
    """Given child counts per group (groups in DFS order), return for each
    child its parent group index and its child index inside the parent."""
    counts = np.asarray(counts, dtype=np.int64)
    total = int(counts.sum())
    parent = np.repeat(np.arange(len(counts), dtype=np.int64), counts)
    starts = np.cumsum(counts) - counts
    cidx = np.arange(total, dtype=np.int64) - np.repeat(starts, counts)
    return parent, cidx


def _leaves_of(level_counts):
    """level_counts[l][g] = number of children of level-l group g.  Returns
    (group_index[l], child_index[l]) per leaf, leaves in DFS order."""
    D = len(level_counts)
    par, cid = [], []
    for l in range(D):
        p, c = _children(level_counts[l])
        par.append(p)
        cid.append(c)
    gidx = [None] * D
    cidx = [None] * D
    gidx[D - 1] = par[D - 1]
    cidx[D - 1] = cid[D - 1]
    for l in range(D - 2, -1, -1):
        g_below = gidx[l + 1]          # index of the leaf's level-(l+1) group
        gidx[l] = par[l][g_below]
        cidx[l] = cid[l][g_below]
    return gidx, cidx


def _last_flags(gidx, cidx):
    """last flag per leaf and level: the leaf's child index at that level is
    the largest child index present in its group (leaves in DFS order, so a
    group's leaves are contiguous)."""
    flags = []
    for g, c in zip(gidx, cidx):
        n = len(g)
        if n == 0:
            flags.append(np.zeros(0, dtype=bool))
            continue
        starts = np.flatnonzero(np.concatenate([[True], g[1:] != g[:-1]]))
        mx = np.maximum.reduceat(c, starts)
        run_len = np.diff(np.concatenate([starts, [n]]))
        flags.append(c == np.repeat(mx, run_len))
    return flags


def _ids(rng, n_groups):
    """A per-level random bijection from group index to a u32 parent_id."""
    a = np.uint64(int(rng.integers(1, 2**31)) * 2 + 1)
    b = np.uint64(int(rng.integers(0, 2**32)))
    idx = np.arange(n_groups, dtype=np.uint64)
    return ((idx * a + b) & _U32).astype(np.uint64)


def stream_from_leaves(name, gidx, cidx, order, lens, rng, *, payload_op, score_op,
                       topk_k, batch, with_score, meta=None):
    """Assemble a Stream from leaves given in DFS order plus an arrival order
    (a permutation of DFS indices)."""
    D = len(gidx)
    flags = _last_flags(gidx, cidx)
    tags = np.empty((D, len(order)), dtype=np.uint64)
    id_tables = [_ids(rng, int(gidx[l].max()) + 1 if len(gidx[l]) else 1) for l in range(D)]

    def level(l):
        tags[l] = pack_tags(id_tables[l][gidx[l][order]], cidx[l][order], flags[l][order])

    with ThreadPoolExecutor(max_workers=D) as ex:
        list(ex.map(level, range(D)))
    lens = np.asarray(lens, dtype=np.int64)[order]
    off = np.zeros(len(order) + 1, dtype=np.int64)
    np.cumsum(lens, out=off[1:])
    payload = _integers(rng, 0, TOKEN_VOCAB, int(off[-1]))
    score = rng.standard_normal(len(order), dtype=np.float32) if with_score else None
    n = len(order)
    nb = n // batch
    sizes = [batch] * nb + ([n - nb * batch] if n - nb * batch else [])
    return Stream(name=name, depth=D, payload_op=tuple(payload_op),
                  score_op=tuple(score_op), topk_k=tuple(topk_k), tags=tags,
                  off=off, payload=payload, score=score,
                  batch_sizes=np.asarray(sizes, dtype=np.int64), meta=meta or {})


def _trim(level_counts, n_leaves):
    """Keep the first n_leaves leaves in DFS order."""
    gidx, cidx = _leaves_of(level_counts)
    return [g[:n_leaves] for g in gidx], [c[:n_leaves] for c in cidx]


def _zipf_capped(rng, n, s=1.2, cap=256):
    k = np.arange(1, cap + 1, dtype=np.float64)
    p = k ** (-s)
    p /= p.sum()
    return rng.choice(np.arange(1, cap + 1), size=n, p=p).astype(np.int64)


def _grow(rng, first_counts, fanout_fns):
    """Level-0 child counts are given; deeper levels draw counts per group."""
    counts = [np.asarray(first_counts, dtype=np.int64)]
    for fn in fanout_fns:
        counts.append(fn(rng, int(counts[-1].sum())))
    return counts


# ----------------------------------------------------------------------------
# the workloads
# ----------------------------------------------------------------------------

def make_tiny(n_leaves=4096, seed=1, n_queries=None, batch=None):
    """Query -> sentence (D=2), CONCAT per query; child order shuffled."""
    rng = np.random.default_rng(seed)
    nq = n_queries if n_queries is not None else n_leaves  # enough queries
    counts = _grow(rng, [nq], [lambda r, n: r.integers(1, 9, size=n)])
    if n_queries is None:
        gidx, cidx = _trim(counts, n_leaves)
    else:
        gidx, cidx = _leaves_of(counts)
    n = len(gidx[0])
    # shuffle queries inside the source and sentences inside each query
    qrank = rng.permutation(int(gidx[1].max()) + 1)
    srank = rng.random(n)
    order = np.lexsort((srank, qrank[gidx[1]]))
    lens = rng.integers(1, 33, size=n)
    return stream_from_leaves(
        "tiny64" if n_queries is not None else "tiny", gidx, cidx, order, lens, rng,
        payload_op=(NONE, CONCAT), score_op=(S_NONE, S_NONE), topk_k=(0, 0),
        batch=batch or n, with_score=False)


def make_factcheck(n_responses=1024, seed=2, batch=65536):
    """response -> claim -> document -> sentence (D=4)."""
    rng = np.random.default_rng(seed)
    counts = _grow(rng, [n_responses], [
        lambda r, n: r.integers(2, 11, size=n),   # claims per response
        lambda r, n: np.full(n, 5, dtype=np.int64),  # documents per claim
        lambda r, n: r.integers(3, 21, size=n),   # sentences per document
    ])
    gidx, cidx = _leaves_of(counts)
    n = len(gidx[0])
    order = rng.permutation(n)
    lens = rng.integers(8, 41, size=n)
    return stream_from_leaves(
        "factcheck", gidx, cidx, order, lens, rng,
        payload_op=(NONE, NONE, NONE, CONCAT), score_op=(S_NONE, S_NONE, S_TOPK, S_MAX),
        topk_k=(0, 0, 3, 0), batch=batch, with_score=True)


def _round_robin_keys(root_of_leaf, rank_in_root, root_sizes, W):
    """Round-robin over W concurrently active roots: each active root emits
    one leaf per round; a finished root's slot goes to the next root."""
    R = len(root_sizes)
    heap = [(0, s) for s in range(min(W, R))]
    start = np.empty(R, dtype=np.int64)
    slot = np.empty(R, dtype=np.int64)
    for r in range(R):
        t, s = heapq.heappop(heap)
        start[r], slot[r] = t, s
        heapq.heappush(heap, (t + int(root_sizes[r]), s))
    return (start[root_of_leaf] + rank_in_root) * W + slot[root_of_leaf]


def _span_fraction(keys, leafparent, batch):
    sk = np.sort(keys)
    pos = np.searchsorted(sk, keys)
    b = pos // batch
    g = leafparent
    G = int(g.max()) + 1
    bmin = np.full(G, np.iinfo(np.int64).max)
    bmax = np.full(G, -1)
    np.minimum.at(bmin, g, b)
    np.maximum.at(bmax, g, b)
    return float(np.mean(bmin != bmax))


def make_throughput(n_leaves=16_000_000, seed=3, batch=1_000_000, target_span=0.20,
                    W=None):
    """Zipf(1.2) fanout capped at 256 (D=4), one source per root."""
    rng = np.random.default_rng(seed)
    n_roots = max(1, int(n_leaves / (26.6 ** 3) * 1.6) + 8)
    while True:
        counts = _grow(rng, np.ones(n_roots, dtype=np.int64), [
            lambda r, n: _zipf_capped(r, n),
            lambda r, n: _zipf_capped(r, n),
            lambda r, n: _zipf_capped(r, n),
        ])
        if counts[3].sum() >= n_leaves:
            break
        n_roots *= 2
    gidx, cidx = _trim(counts, n_leaves)
    n = len(gidx[0])
    root = gidx[0]
    R = int(root.max()) + 1
    root_sizes = np.bincount(root, minlength=R)
    # random order of leaves inside each root
    u = rng.integers(0, 2**32, size=n, dtype=np.uint64)
    within = np.argsort((root.astype(np.uint64) << np.uint64(32)) | u, kind="stable")
    rank_in_root = np.empty(n, dtype=np.int64)
    rstart = np.cumsum(root_sizes) - root_sizes
    rank_in_root[within] = np.arange(n, dtype=np.int64) - rstart[root[within]]
    leafparent = gidx[3]
    if W is None:
        lo, hi = 1, max(1, R)
        f_hi = _span_fraction(_round_robin_keys(root, rank_in_root, root_sizes, hi),
                              leafparent, batch)
        W = hi
        if f_hi > target_span:
            for _ in range(40):
                if hi - lo <= 1:
                    break
                mid = (lo + hi) // 2
                f = _span_fraction(_round_robin_keys(root, rank_in_root, root_sizes, mid),
                                   leafparent, batch)
                if f < target_span:
                    lo = mid
                else:
                    hi = mid
            f_lo = _span_fraction(_round_robin_keys(root, rank_in_root, root_sizes, lo),
                                  leafparent, batch)
            f_hi = _span_fraction(_round_robin_keys(root, rank_in_root, root_sizes, hi),
                                  leafparent, batch)
            W = lo if abs(f_lo - target_span) <= abs(f_hi - target_span) else hi
    keys = _round_robin_keys(root, rank_in_root, root_sizes, W)
    order = np.argsort(keys, kind="stable")
    frac = _span_fraction(keys, leafparent, batch)
    lens = rng.integers(1, 65, size=n)
    return stream_from_leaves(
        "throughput", gidx, cidx, order, lens, rng,
        payload_op=(NONE, NONE, NONE, CONCAT), score_op=(S_NONE,) * 4, topk_k=(0,) * 4,
        batch=batch, with_score=False, meta=dict(window=int(W), span_fraction=frac))


def make_tokens(n_streams=4096, tokens_per_stream=24414, seed=4, batch=8192):
    """Token-granularity streams (D=2), single-token leaves, round-robin with
    seeded jitter."""
    rng = np.random.default_rng(seed)
    counts = [np.array([n_streams], dtype=np.int64),
              np.full(n_streams, tokens_per_stream, dtype=np.int64)]
    gidx, cidx = _leaves_of(counts)
    s = gidx[1]
    t = cidx[1]
    u = rng.random(len(s))
    key = t * n_streams + s + np.floor(n_streams * u).astype(np.int64)
    order = np.argsort(key, kind="stable")
    lens = np.ones(len(s), dtype=np.int64)
    return stream_from_leaves(
        "tokens", gidx, cidx, order, lens, rng,
        payload_op=(NONE, CONCAT), score_op=(S_NONE, S_NONE), topk_k=(0, 0),
        batch=batch, with_score=False)


def make_adversarial(n_leaves=64 * 2**20, hot_leaves=2**20, seed=5, batch=2 * 2**20,
                     max_shift=3):
    """D=6 long tail of fanout U{1..4} plus one hot leaf-parent; the subtree
    of every group's last-flagged child arrives up to max_shift batches early."""
    rng = np.random.default_rng(seed)
    n_tail = n_leaves - hot_leaves
    n_roots = max(1, int(n_tail / 2.5 ** 5 * 1.3) + 4)
    f14 = lambda r, n: r.integers(1, 5, size=n)  # noqa: E731
    while True:
        counts = _grow(rng, np.ones(n_roots, dtype=np.int64), [f14] * 5)
        if counts[5].sum() >= n_tail:
            break
        n_roots *= 2
    tg, tc = _trim(counts, n_tail)
    # the hot chain: its own group at every level above, with one leaf parent of hot_leaves
    hot_counts = [np.ones(1, dtype=np.int64)] * 5 + [np.array([hot_leaves], dtype=np.int64)]
    hg, hc = _leaves_of(hot_counts)
    D = 6
    gidx, cidx = [], []
    for l in range(D):
        base = int(tg[l].max()) + 1 if n_tail else 0
        gidx.append(np.concatenate([tg[l], hg[l] + base]))
        cidx.append(np.concatenate([tc[l], hc[l]]))
    n = n_tail + hot_leaves
    flags = _last_flags(gidx, cidx)
    # per-group shift (in batches) for the last-flagged child's subtree
    shift = np.zeros(n, dtype=np.int64)
    for l in range(D):
        G = int(gidx[l].max()) + 1
        s_g = rng.integers(0, max_shift + 1, size=G)
        cand = np.where(flags[l], s_g[gidx[l]], 0)
        np.maximum(shift, cand, out=shift)
    scale = n / max(1, n_tail)
    key = np.empty(n, dtype=np.float64)
    key[:n_tail] = np.arange(n_tail, dtype=np.float64) * scale - shift[:n_tail] * batch
    np.maximum(key, 0.0, out=key)
    key[n_tail:] = rng.random(hot_leaves) * n
    order = np.argsort(key, kind="stable")
    lens = rng.integers(1, 17, size=n)
    return stream_from_leaves(
        "adversarial", gidx, cidx, order, lens, rng,
        payload_op=(NONE,) * 5 + (CONCAT,), score_op=(S_NONE,) * 5 + (S_TOPK,),
        topk_k=(0,) * 5 + (8,), batch=batch, with_score=True)


def make_tot(n_queries=2048, seed=7, batch=65536, iters=3, keep=5, thoughts=(30, 50), evals=3):
    """Tree-of-Thoughts shaped (Sec. 6.1.2): each query runs `iters`
    iterations; in iteration i every frontier node (the query itself, then
    the `keep` best thoughts of each node of the previous iteration: 1, 5, 25
    nodes) expands into U{30..50} thoughts, and every thought is evaluated
    `evals` times (the leaves, each with an fp32 score and U{1..16} tokens).
    Tags, D=3: level 0 = the query's iteration (children: its frontier
    nodes), level 1 = a frontier node (children: its thoughts; TOPK(keep) by
    score), level 2 = a thought (children: its evaluations; MAX of the
    scores, CONCAT of their texts).  Queries start at staggered times; a
    query's iteration i+1 arrives after its iteration i, and fragments are
    shuffled within each iteration's window."""
    rng = np.random.default_rng(seed)
    fan = [keep ** i for i in range(iters)]                     # frontier nodes per iteration
    it_counts = np.tile(np.asarray(fan, dtype=np.int64), n_queries)  # level-0 groups: (query, iter)
    counts = _grow(rng, it_counts, [
        lambda r, n: r.integers(thoughts[0], thoughts[1] + 1, size=n),
        lambda r, n: np.full(n, evals, dtype=np.int64)])
    gidx, cidx = _leaves_of(counts)
    n = len(gidx[0])
    g0 = gidx[0]                                   # level-0 group = query * iters + iteration
    q, it = g0 // iters, g0 % iters
    start = rng.random(n_queries) * iters          # query start, in iteration windows
    key = start[q] + it + rng.random(n) * 0.999
    order = np.argsort(key, kind="stable")
    lens = rng.integers(1, 17, size=n)
    return stream_from_leaves(
        "tot", gidx, cidx, order, lens, rng,
        payload_op=(NONE, NONE, CONCAT), score_op=(S_NONE, S_TOPK, S_MAX), topk_k=(0, keep, 0),
        batch=batch, with_score=True, meta={"iters": iters, "keep": keep})


@dataclass
class SplitInput:
    """Token streams for split_text: streams x tokens, sentences of U{1..max_sentence}
    tokens each closed by one of the delimiter ids, plus each stream's own tags
    (one level: child s of a single source) and its id at the new level."""
    tok_off: np.ndarray    # int64 [n_src + 1]
    tokens: np.ndarray     # int32
    delims: tuple
    src_tags: np.ndarray   # uint64 [1, n_src]
    src_id: np.ndarray     # uint32 [n_src]


def make_split_input(n_streams=4096, tokens_per_stream=24414, seed=8, delims=(198, 13), max_sentence=64,
                     empty_every=0):
    rng = np.random.default_rng(seed)
    lens = np.full(n_streams, tokens_per_stream, dtype=np.int64)
    if empty_every:
        lens[::empty_every] = 0
    n = int(lens.sum())
    tokens = _integers(rng, 0, TOKEN_VOCAB, n).astype(np.int32)
    # ordinary tokens never collide with a delimiter id
    dl = np.asarray(delims, dtype=np.int32)
    hit = np.isin(tokens, dl)
    tokens[hit] = (tokens[hit] + 1) % TOKEN_VOCAB
    # a delimiter closes every sentence
    gaps = rng.integers(1, max_sentence + 1, size=n // 1 + 1)
    ends = np.cumsum(gaps) - 1
    ends = ends[ends < n]
    tokens[ends] = dl[rng.integers(0, len(dl), size=len(ends))]
    tok_off = np.concatenate([[0], np.cumsum(lens)]).astype(np.int64)
    src_tags = pack_tags(np.full(n_streams, 9, dtype=np.uint64), np.arange(n_streams, dtype=np.uint64),
                         (np.arange(n_streams) == n_streams - 1).astype(np.uint64))[None, :]
    src_id = (rng.permutation(n_streams) + 1000).astype(np.uint32)
    return SplitInput(tok_off=tok_off, tokens=tokens, delims=tuple(int(x) for x in delims),
                      src_tags=np.ascontiguousarray(src_tags), src_id=src_id)


def make_stream(name: str, small: bool = False) -> Stream:
    """Full-size stream by name, or a scaled-down stream of the same shape
    (``small=True``) that the CPU oracle finishes in seconds and that still
    spans several batches."""
    if name == "tiny":
        return make_tiny()
    if name == "tiny64":
        return make_tiny(n_queries=64, seed=6)
    if name == "factcheck":
        return make_factcheck(n_responses=48, batch=4096) if small else make_factcheck()
    if name == "throughput":
        # W=5 is what the bisection picks for seed 3 at full size (18.3% of the
        # leaf-parent groups span a batch boundary); pinned to skip the search
        return (make_throughput(n_leaves=200_000, batch=16_384) if small
                else make_throughput(W=5))
    if name == "tokens":
        return (make_tokens(n_streams=256, tokens_per_stream=300, batch=1024) if small
                else make_tokens())
    if name == "adversarial":
        return (make_adversarial(n_leaves=3 * 2**16, hot_leaves=2**14, batch=2**14)
                if small else make_adversarial())
    if name == "tot":
        return make_tot(n_queries=12, batch=4096) if small else make_tot()
    raise ValueError(f"unknown stream {name!r}; one of {CONFIG_NAMES}")
