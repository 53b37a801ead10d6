"""Streaming release with the CONCAT level above the leaf parent, on the GPU,
bit for bit against the oracle through the C ABI.

Sec. 3.2: each pmap puts its outputs back in order and passes them on as a
stream; a CONCAT level M < D-1 reconstitutes a stream whose items are its
children's concatenations.  With streaming release, after every batch an open
level-M group whose run of complete children grew emits those children as a
partial record, and its final record carries the rest.  Here the children of
a level-M group are groups themselves, which complete in any order and hand
their concatenations up as spans.  The cases: the workloads with CONCAT moved
up (including TOPK at the CONCAT level), drained every batch and every third;
depth-3 streams whose level-2 groups complete out of order, by blocks and in
reverse (buffered spans kept in part and moved down, spans across arena
chunks); random small trees with every CONCAT level above the leaf parent, in
random orders and batch cuts; and the arena back to empty at the stream's end.
"""
import dataclasses
import random

import numpy as np
import pytest

torch = pytest.importorskip("torch")

import paper_2403_04311_gb300 as alto
from fragments import split, to_batch, tree_fragments
from gen import make_stream
from gen.streams import Stream
from gpu_harness import assert_same, run_both_stream, run_gpu_batches, run_oracle_batches, stream_caps

pytestmark = pytest.mark.gpu


def _with_concat_at(s, m):
    po = [0] * s.depth
    po[m] = 1
    return dataclasses.replace(s, payload_op=tuple(po))


def _caps(s):
    # children of every level may take dense slots in one batch, and a leaf's
    # tokens may sit in two levels' vectors while they are handed up
    caps = stream_caps(s, arena_factor=6, stream_release=True)
    caps["max_emit_children"] = s.n * s.depth + 16
    return caps


def _check(s, drain_every=1):
    o, g = run_both_stream(s, drain_every=drain_every, caps=_caps(s), stream_release=True)
    assert all(d.status == 0 for d in o)
    assert_same(o, g, f"{s.name} {s.payload_op}/{drain_every}")
    return sum(int(((d.records["ops"] & 0x80) != 0).sum()) for d in o)


# (a root of the throughput stream has one child, and the tiny stream is one
# batch: those two release nothing, the others do)
@pytest.mark.parametrize("name,m,releases", [("throughput", 0, False), ("throughput", 1, True),
                                             ("throughput", 2, True), ("factcheck", 1, True),
                                             ("factcheck", 2, True), ("tot", 1, True),
                                             ("adversarial", 2, True), ("adversarial", 4, True),
                                             ("tiny", 0, False)])
@pytest.mark.parametrize("drain_every", [1, 3])
def test_workloads_stream_release_above_leaf_parent(name, m, releases, drain_every):
    s = _with_concat_at(make_stream(name, small=True), m)
    n_part = _check(s, drain_every)
    assert (n_part > 0) == releases


def _pack(p, c, last):
    return (np.asarray(p, np.uint64) << np.uint64(32)) | (np.asarray(last, np.uint64) << np.uint64(31)) | \
        np.asarray(c, np.uint64)


def _spans_stream(n_groups, n_children, leaves, max_len, order, batch, seed):
    """Depth 3: one source (level 0), n_groups streams (level 1, CONCAT) of
    n_children pieces (level 2), each piece `leaves` leaves.  A piece's leaves
    arrive together, so pieces complete in the order `order(rng, n)` gives;
    streams are interleaved at random."""
    rng = np.random.default_rng(seed)
    queues = [list(order(rng, n_children)) for _ in range(n_groups)]
    live = list(range(n_groups))
    rows = []
    while live:
        k = int(rng.integers(0, len(live)))
        g = live[k]
        c = queues[g].pop(0)
        for j in rng.permutation(leaves):
            rows.append((g, c, int(j)))
        if not queues[g]:
            live.pop(k)
    g_of = np.asarray([r[0] for r in rows], np.int64)
    c_of = np.asarray([r[1] for r in rows], np.int64)
    j_of = np.asarray([r[2] for r in rows], np.int64)
    n = len(rows)
    tags = np.zeros((3, n), np.uint64)
    tags[0] = _pack(1, g_of, g_of == n_groups - 1)
    tags[1] = _pack(1000 + g_of, c_of, c_of == n_children - 1)
    tags[2] = _pack(100000 + g_of * n_children + c_of, j_of, j_of == leaves - 1)
    lens = rng.integers(0, max_len + 1, size=n)
    off = np.concatenate([[0], np.cumsum(lens)]).astype(np.int64)
    payload = rng.integers(0, 1 << 30, size=int(off[-1])).astype(np.int32)
    sizes = [batch] * (n // batch) + ([n % batch] if n % batch else [])
    return Stream(name="spans", depth=3, payload_op=(0, 1, 0), score_op=(0, 0, 0), topk_k=(0, 0, 0),
                  tags=tags, off=off, payload=payload, score=None, batch_sizes=np.asarray(sizes), meta={})


def _blocks(rng, n):
    """Blocks of 50 pieces in a shuffled block order, in order inside a block."""
    nb = (n + 49) // 50
    out = []
    for b in rng.permutation(nb):
        out.extend(range(50 * b, min(50 * (b + 1), n)))
    return out


@pytest.mark.parametrize("order,max_len,batch,releases", [
    (_blocks, 12, 96, True),                               # backlogs kept in part and moved down
    (_blocks, 150, 131, True),                             # spans across arena chunks
    (lambda rng, n: list(range(n))[::-1], 6, 64, False),   # everything buffered until piece 0
    (lambda rng, n: list(rng.permutation(n)), 9, 200, True),
])
def test_pieces_complete_out_of_order(order, max_len, batch, releases):
    s = _spans_stream(12, 300, 3, max_len, order, batch, seed=max_len + batch)
    n_part = _check(s, 1)
    assert (n_part > 0) == releases
    _check(s, 4)


def _shapes(depth):
    if depth == 1:
        return [1, 2, 3]
    sub = _shapes(depth - 1)
    return [[a] for a in sub] + [[a, b] for a in sub for b in sub][:6]


@pytest.mark.parametrize("depth", [2, 3])
def test_small_trees_concat_above_leaf_parent(depth):
    rng = random.Random(40 + depth)
    cases = 0
    for shape in _shapes(depth):
        frags = tree_fragments(shape, score_fn=lambda k: float(k % 5))
        n = len(frags)
        for m in range(depth - 1):
            po = [0] * depth
            po[m] = 1
            for _ in range(8):
                p = list(range(n))
                rng.shuffle(p)
                cuts = sorted(rng.sample(range(1, n), min(n - 1, rng.randint(0, 3)))) if n > 1 else []
                sizes = [b - a for a, b in zip([0] + cuts, cuts + [n])]
                batches = [to_batch(part, depth, False) for part in split([frags[i] for i in p], sizes)]
                caps = dict(max_batch_fragments=n, max_batch_payload=max(1, sum(len(f[1]) for f in frags)),
                            max_open_groups=256, arena_elems=1 << 13, out_records=256,
                            out_payload_elems=1 << 10, out_topk=64, max_emit_children=256,
                            stream_release=True)
                _, g = run_gpu_batches(depth, po, [0] * depth, [0] * depth, batches, caps)
                o = run_oracle_batches(depth, po, [0] * depth, [0] * depth, batches, stream_release=True)
                assert_same(o, g, f"{shape} M={m} {p} {sizes}")
                cases += 1
    assert cases >= 40


def test_arena_returns_to_empty_with_releases():
    """Every group completes by the end of the stream: after the partial
    releases moved the buffers down, every chunk is back on the free stacks."""
    s = _spans_stream(6, 200, 2, 20, _blocks, 77, seed=5)
    agg = alto.Aggregator(s.depth, s.payload_op, s.score_op, s.topk_k, stream_release=True, **_caps(s))
    partial = 0
    for b in range(s.n_batches):
        db = alto.to_device(s.batch(b))
        assert agg.push(db.tags, db.off, db.payload, db.score) == alto.OK
        d = agg.drain()
        assert d.status == alto.OK
        rec, _, _ = d.host()
        partial += int(((rec["ops"] & 0x80) != 0).sum())
    st, open_groups, arena_used = agg.stats()
    agg.close()
    assert partial > 0
    assert st == alto.OK and open_groups == 0 and arena_used == 0
