"""Streaming release on the GPU against the oracle, bit for bit, through the C ABI.

Sec. 3.2: the outputs of a pmap are put back in order and passed on as a
stream.  With streaming release, after every batch an open CONCAT group
(leaf-parent level) emits the run of present children that follows what it
released before; the final record carries the rest.  The cases: the seven
workloads; groups whose children arrive out of order, by blocks (backlogs
that are kept in part and moved down in their buffers) or by a local shuffle
(many short releases); leaves long enough that spans cross arena chunks; TOPK
at the leaf parent; random small trees in every arrival order and batch cut;
and a released child given again (EDUP).
"""
import random

import numpy as np
import pytest

torch = pytest.importorskip("torch")

import paper_2403_04311_gb300 as alto
from fragments import split, to_batch, tree_fragments
from gen import make_stream
from gen.streams import Stream
from gpu_harness import assert_same, run_both_stream, run_gpu_batches, run_oracle_batches

pytestmark = pytest.mark.gpu


def _pack(p, c, last):
    return (np.asarray(p, np.uint64) << np.uint64(32)) | (np.asarray(last, np.uint64) << np.uint64(31)) | \
        np.asarray(c, np.uint64)


def _groups_stream(n_groups, n_children, max_len, order_fn, batch, seed, topk=False):
    """Depth 2: one source (level 0) with n_groups streams (level 1) of
    n_children pieces each; order_fn(rng, n_children) gives each stream's
    arrival order of child indices; streams are interleaved at random."""
    rng = np.random.default_rng(seed)
    g_of, c_of = [], []
    queues = [list(order_fn(rng, n_children)) for _ in range(n_groups)]
    live = list(range(n_groups))
    while live:
        k = int(rng.integers(0, len(live)))
        g = live[k]
        g_of.append(g)
        c_of.append(queues[g].pop(0))
        if not queues[g]:
            live.pop(k)
    g_of = np.asarray(g_of, np.int64)
    c_of = np.asarray(c_of, np.int64)
    n = len(g_of)
    tags = np.zeros((2, n), np.uint64)
    tags[0] = _pack(1, g_of, g_of == n_groups - 1)
    tags[1] = _pack(1000 + g_of, c_of, c_of == n_children - 1)
    lens = rng.integers(0, max_len + 1, size=n)
    off = np.concatenate([[0], np.cumsum(lens)]).astype(np.int64)
    payload = rng.integers(0, 1 << 30, size=int(off[-1])).astype(np.int32)
    score = rng.standard_normal(n).astype(np.float32) if topk else None
    sizes = [batch] * (n // batch) + ([n % batch] if n % batch else [])
    return Stream(name="groups", depth=2, payload_op=(0, 1), score_op=(0, 2 if topk else 0),
                  topk_k=(0, 3 if topk else 0), tags=tags, off=off, payload=payload, score=score,
                  batch_sizes=np.asarray(sizes), meta={})


def _blocks(rng, n):
    """Blocks of 100 children in a shuffled block order, in order inside a block."""
    nb = (n + 99) // 100
    out = []
    for b in rng.permutation(nb):
        out.extend(range(100 * b, min(100 * (b + 1), n)))
    return out


def _local(rng, n, w=16):
    """In order up to a shuffle inside windows of w."""
    out = []
    for s in range(0, n, w):
        out.extend(list(s + rng.permutation(min(w, n - s))))
    return out


def _check(s, drain_every=1):
    o, g = run_both_stream(s, drain_every=drain_every, stream_release=True)
    assert all(d.status == 0 for d in o)
    assert_same(o, g, f"{s.name}/{drain_every}")
    n_part = sum(int(((d.records["ops"] & 0x80) != 0).sum()) for d in o)
    return n_part


@pytest.mark.parametrize("name", ["tiny", "tiny64", "factcheck", "throughput", "tokens", "adversarial", "tot"])
@pytest.mark.parametrize("drain_every", [1, 3])
def test_workloads_stream_release(name, drain_every):
    s = make_stream(name, small=True)
    n_part = _check(s, drain_every)
    assert n_part > 0 or s.n_batches == 1


@pytest.mark.parametrize("order,max_len,batch", [
    (_blocks, 40, 64),       # backlogs kept in part and moved down
    (_blocks, 300, 97),      # spans across arena chunks
    (_local, 20, 500),       # many short releases
    (lambda rng, n: list(range(n))[::-1], 10, 128),   # everything buffered until child 0
])
def test_out_of_order_streams(order, max_len, batch):
    s = _groups_stream(24, 700, max_len, order, batch, seed=max_len + batch)
    _check(s, 1)
    _check(s, 4)


def test_topk_leaf_parent_with_stream_release():
    s = _groups_stream(40, 300, 12, _local, 256, seed=5, topk=True)
    assert _check(s, 1) > 0


def test_hand_worked_stream():
    def f(c, last=False):
        return (((1, 0, True), (9, c, last)), [10 * c, 10 * c + 1], 0.0)
    frags = [f(1), f(0), f(3, True), f(2)]
    batches = [to_batch(p, 2, False) for p in split(frags, [2, 1, 1])]
    caps = dict(max_batch_fragments=4, max_batch_payload=8, max_open_groups=64, arena_elems=1 << 12,
                out_records=64, out_payload_elems=64, out_topk=16, max_emit_children=64,
                stream_release=True)
    _, g = run_gpu_batches(2, [0, 1], [0, 0], [0, 0], batches, caps)
    o = run_oracle_batches(2, [0, 1], [0, 0], [0, 0], batches, stream_release=True)
    assert_same(o, g, "hand-worked")
    st, rec, pay, _ = g[0]
    assert [(int(r["n_children"]), int(r["ops"])) for r in rec] == [(2, 0x81)]
    assert pay.tolist() == [0, 1, 10, 11]
    assert len(g[1][1]) == 0
    st, rec, pay, _ = g[2]
    assert [(int(r["level"]), int(r["n_children"]), int(r["ops"])) for r in rec] == [(1, 4, 1), (0, 1, 0)]
    assert pay.tolist() == [20, 21, 30, 31]


def _shapes(depth):
    if depth == 1:
        return [1, 2, 3, 5]
    sub = _shapes(depth - 1)
    return [[a] for a in sub] + [[a, b] for a in sub for b in sub][:6]


@pytest.mark.parametrize("depth", [1, 2, 3])
def test_small_trees_every_order(depth):
    rng = random.Random(depth)
    cases = 0
    for shape in _shapes(depth):
        frags = tree_fragments(shape, score_fn=lambda k: float(k % 5))
        n = len(frags)
        po = [0] * depth
        po[-1] = 1
        for _ in range(12):
            p = list(range(n))
            rng.shuffle(p)
            cuts = sorted(rng.sample(range(1, n), min(n - 1, rng.randint(0, 3)))) if n > 1 else []
            sizes = [b - a for a, b in zip([0] + cuts, cuts + [n])]
            batches = [to_batch(part, depth, False) for part in split([frags[i] for i in p], sizes)]
            caps = dict(max_batch_fragments=n, max_batch_payload=max(1, sum(len(f[1]) for f in frags)),
                        max_open_groups=256, arena_elems=1 << 12, out_records=256, out_payload_elems=1 << 10,
                        out_topk=64, max_emit_children=256, stream_release=True)
            _, g = run_gpu_batches(depth, po, [0] * depth, [0] * depth, batches, caps)
            o = run_oracle_batches(depth, po, [0] * depth, [0] * depth, batches, stream_release=True)
            assert_same(o, g, f"{shape} {p} {sizes}")
            cases += 1
    assert cases >= 40


def test_released_child_again_is_edup():
    def f(c, last=False):
        return (((1, 0, True), (9, c, last)), [c], 0.0)
    batches = [to_batch([f(0), f(1)], 2, False), to_batch([f(1)], 2, False)]
    caps = dict(max_batch_fragments=4, max_batch_payload=8, max_open_groups=64, arena_elems=1 << 12,
                out_records=64, out_payload_elems=64, out_topk=16, max_emit_children=64,
                stream_release=True)
    pushes, g = run_gpu_batches(2, [0, 1], [0, 0], [0, 0], batches, caps)
    o = run_oracle_batches(2, [0, 1], [0, 0], [0, 0], batches, stream_release=True)
    assert o[0].status == 0 and o[1].status == alto.EDUP
    assert g[0][0] == alto.OK and g[1][0] == alto.EDUP



@pytest.mark.slow
def test_stream_release_fullsize_throughput():
    """The 16M-fragment throughput stream with streaming release, the bench's
    capacities: the first two batches bit for bit against the oracle; over the
    whole run, every leaf-parent group's partial records grow strictly and end
    in one final record with n_children = last + 1, the records of every drain
    are in strictly increasing (seq, deeper first) order, and for a seeded
    sample of groups the released payloads, in record order, are the group's
    leaves in child order."""
    import bench
    import oracle
    s = make_stream("throughput")
    D = s.depth
    caps = bench.stream_caps(s, stream_release=True)
    agg = alto.Aggregator(s.depth, s.payload_op, s.score_op, s.topk_k, **caps)
    o = oracle.Oracle.for_stream(s, stream_release=True)
    leaf_pid = (s.tags[D - 1] >> np.uint64(32)).astype(np.int64)
    rng = np.random.default_rng(11)
    sample = set(rng.choice(np.unique(leaf_pid), size=128, replace=False).tolist())
    got_pay = {p: [] for p in sample}
    pids, counts = np.unique(leaf_pid, return_counts=True)
    n_leaves = dict(zip(pids.tolist(), counts.tolist()))
    last_n, finals = {}, 0
    for b in range(s.n_batches):
        bt = s.batch(b)
        db = alto.to_device(bt)
        assert agg.push(db.tags, db.off, db.payload, db.score) == alto.OK
        d = agg.drain()
        assert d.status == alto.OK, b
        rec, pay, _ = d.host()
        if b < 2:
            o.push_batch(bt)
            od = o.drain()
            assert np.array_equal(rec.view(np.uint8), od.records.view(np.uint8)), b
            assert np.array_equal(pay, od.payload), b
        keys = rec["completion_seq"].astype(np.int64) * 16 - rec["level"].astype(np.int64)
        assert np.all(np.diff(keys) > 0), b
        m = rec["level"] == D - 1
        for r in rec[m]:
            p, n_ch = int(r["parent_id"]), int(r["n_children"])
            assert n_ch > last_n.get(p, 0), (b, p)
            if int(r["ops"]) & 0x80:
                last_n[p] = n_ch
            else:
                assert n_ch == n_leaves[p], (b, p)
                last_n[p] = 1 << 40       # nothing may follow the final record
                finals += 1
            if p in sample:
                got_pay[p].extend(pay[int(r["payload_off"]):int(r["payload_off"]) + int(r["payload_len"])].tolist())
        del db
    agg.close()
    o.close()
    assert finals == len(pids)
    leaf_c = (s.tags[D - 1] & np.uint64(0x7FFFFFFF)).astype(np.int64)
    for p in sample:
        idx = np.flatnonzero(leaf_pid == p)
        idx = idx[np.argsort(leaf_c[idx], kind="stable")]
        want = np.concatenate([s.payload[s.off[i]:s.off[i + 1]] for i in idx]).tolist()
        assert got_pay[p] == want, p


def test_stream_release_on_a_segment_longer_than_a_warp_share():
    """One group of 20,000 children in blocks of 1,000 in shuffled block order,
    8,192-fragment batches: its segment in a batch is longer than 4,096 leaves
    (the block-wide reduce), and releases both take leaves straight from the
    batch and drop buffered ones."""
    s = _groups_stream(1, 20_000, 6, lambda rng, n: [c for b in rng.permutation(n // 1000)
                                                       for c in range(1000 * b, 1000 * (b + 1))], 8192, seed=3)
    assert _check(s, 1) > 0
