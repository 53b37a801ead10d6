"""Oracle pinned to library routines and invariants.

* depth 1, one batch: the CONCAT payload is the leaves stably sorted by child
  index (numpy argsort);
* one batch, CONCAT at level 0 of a deeper tree: the leaves in lexicographic
  child-index-path order (numpy lexsort);
* TOPK: numpy lexsort on (child index, -totalOrder key); MAX: numpy max of
  totalOrder keys;
* on every generated workload (small variants): each record's completion
  seq is the largest arrival index in its subtree, records come in
  (seq, deeper level first) order, every group is emitted once and after all
  of its descendants, n_children is the number of distinct children, the
  CONCAT payload is the subtree's leaves in path order, and the pushed payload
  is conserved."""
import numpy as np
import pytest

import oracle
from gen import CONCAT, make_stream, pack_tags
from gen.streams import Stream


def total_order_keys(x):
    u = np.asarray(x, dtype=np.float32).view(np.uint32).astype(np.uint64)
    neg = (u & 0x80000000) != 0
    return np.where(neg, u ^ 0xFFFFFFFF, u | 0x80000000)


def one_group_stream(n, seed, with_score):
    rng = np.random.default_rng(seed)
    c = rng.permutation(n)
    tags = pack_tags(np.full(n, 77), c, c == n - 1)[None, :]
    lens = rng.integers(0, 5, size=n)
    off = np.concatenate([[0], np.cumsum(lens)])
    pay = rng.integers(-1000, 1000, size=int(off[-1]), dtype=np.int32)
    sc = rng.choice(np.array([-2.0, -0.0, 0.0, 1.0, 1.0, 3.0], np.float32), size=n) if with_score else None
    return c, tags, off, pay, sc


def test_depth1_concat_is_stable_sort_by_child_index():
    c, tags, off, pay, _ = one_group_stream(500, 1, False)
    o = oracle.Oracle(1, [1], [0], [0])
    o.push(tags, off.astype(np.uint32), pay)
    d = o.drain()
    assert d.status == 0 and len(d.records) == 1
    order = np.argsort(c, kind="stable")
    want = np.concatenate([pay[off[i]:off[i + 1]] for i in order])
    assert np.array_equal(d.payload, want)
    assert d.records[0]["n_children"] == 500 and d.records[0]["completion_seq"] == 499


@pytest.mark.parametrize("k", [1, 3, 8, 32])
def test_topk_and_max_are_lexsort_selection(k):
    c, tags, off, pay, sc = one_group_stream(300, 2 + k, True)
    o = oracle.Oracle(1, [0], [2], [k])
    o.push(tags, off.astype(np.uint32), pay, sc)
    d = o.drain()
    keys = total_order_keys(sc).astype(np.int64)
    sel = np.lexsort((c, -keys))[:k]
    assert [int(p["child_index"]) for p in d.topk] == c[sel].tolist()
    assert np.array_equal(np.array([p["score"] for p in d.topk], np.float32).view(np.uint32),
                          sc[sel].view(np.uint32))
    best = sc[np.argmax(keys)]
    assert np.float32(d.records[0]["score"]).view(np.uint32) == best.view(np.uint32)
    o2 = oracle.Oracle(1, [0], [1], [0])
    o2.push(tags, off.astype(np.uint32), pay, sc)
    d2 = o2.drain()
    assert np.float32(d2.records[0]["score"]).view(np.uint32) == best.view(np.uint32)
    assert len(d2.topk) == 0


def test_single_batch_level0_concat_is_lexsort_of_paths():
    s = make_stream("factcheck", small=True)
    o = oracle.Oracle(s.depth, [CONCAT, 0, 0, 0], [0] * 4, [0] * 4)
    n = s.n
    o.push(s.tags, s.off.astype(np.uint32), s.payload, None)
    d = o.drain()
    assert d.status == 0
    top = [r for r in d.records if r["level"] == 0]
    assert len(top) == 1 and top[0]["payload_len"] == s.payload.size
    cs = [(s.tags[l] & np.uint64(0x7FFFFFFF)).astype(np.int64) for l in range(s.depth)]
    order = np.lexsort(tuple(reversed(cs)))
    want = np.concatenate([s.payload[s.off[i]:s.off[i + 1]] for i in order])
    assert np.array_equal(d.payload, want)
    assert top[0]["completion_seq"] == n - 1


def group_table(s: Stream):
    """Independent per-group facts from the stream arrays: for each (level,
    parent id): arrival indices of its leaves and its distinct children."""
    D, n = s.depth, s.n
    pid = [(s.tags[l] >> np.uint64(32)).astype(np.int64) for l in range(D)]
    cid = [(s.tags[l] & np.uint64(0x7FFFFFFF)).astype(np.int64) for l in range(D)]
    facts = {}
    seq = np.arange(n)
    for l in range(D):
        order = np.argsort(pid[l], kind="stable")
        p_sorted = pid[l][order]
        starts = np.flatnonzero(np.concatenate([[True], p_sorted[1:] != p_sorted[:-1]]))
        ends = np.concatenate([starts[1:], [n]])
        for a, b in zip(starts, ends):
            idx = order[a:b]
            facts[(l, int(p_sorted[a]))] = dict(
                max_seq=int(seq[idx].max()), n_children=len(np.unique(cid[l][idx])),
                leaves=idx)
    return facts, pid, cid


@pytest.mark.parametrize("name", ["tiny", "tiny64", "factcheck", "throughput", "tokens", "adversarial", "tot"])
def test_invariants_on_workloads(name):
    s = make_stream(name, small=True)
    drains = oracle.run_stream(s, drain_every=2)
    drains2 = oracle.run_stream(s, drain_every=2)
    assert all(d.status == 0 for d in drains)
    facts, pid, cid = group_table(s)
    recs = np.concatenate([d.records for d in drains])
    # determinism
    assert np.array_equal(recs, np.concatenate([d.records for d in drains2]))
    # every group emitted exactly once (all streams complete by the end)
    keys = list(zip(recs["level"].tolist(), recs["parent_id"].tolist()))
    assert len(keys) == len(set(keys)) == len(facts)
    # order: (completion seq asc, level desc), strictly
    cs = recs["completion_seq"].astype(np.int64)
    lv = recs["level"].astype(np.int64)
    comp = cs * 16 + (15 - lv)
    assert np.all(np.diff(comp) > 0)
    pos = {k: i for i, k in enumerate(keys)}
    for (l, p), f in facts.items():
        r = recs[pos[(l, p)]]
        assert int(r["completion_seq"]) == f["max_seq"]
        assert int(r["n_children"]) == f["n_children"]
        if l > 0:
            # parent after every descendant
            i = f["leaves"][0]
            parent = (l - 1, int(pid[l - 1][i]))
            assert pos[parent] > pos[(l, p)]
    # CONCAT payload: the subtree's leaves in path order, and conservation
    m = [l for l in range(s.depth) if s.payload_op[l] == CONCAT]
    if m:
        M = m[0]
        total = 0
        for d in drains:
            for r in d.records[d.records["level"] == M]:
                f = facts[(M, int(r["parent_id"]))]
                idx = f["leaves"]
                order = np.lexsort(tuple(cid[l][idx] for l in reversed(range(M, s.depth))))
                want = np.concatenate([s.payload[s.off[i]:s.off[i + 1]] for i in idx[order]])
                got = d.payload[int(r["payload_off"]):int(r["payload_off"]) + int(r["payload_len"])]
                assert np.array_equal(got, want)
                total += int(r["payload_len"])
        assert total == s.payload.size


def _empty(s):
    return dict(n=0, seq_base=0, tags=np.zeros((s.depth, 0), np.uint64), off=np.zeros(1, np.uint32),
                payload=np.zeros(0, np.int32), score=None if s.score is None else np.zeros(0, np.float32))


@pytest.mark.parametrize("name", ["tiny", "factcheck", "throughput", "adversarial", "tot"])
@pytest.mark.parametrize("stream_release", [False, True])
def test_empty_batches_change_nothing(name, stream_release):
    """An empty batch brings no fragment, so no group changes (Sec. 3.1: only
    a delimiter closes a stream): with empty batches before, between and
    after the stream's batches, the drains after the empty ones hold
    nothing and the others equal the run without them."""
    s = make_stream(name, small=True)
    plain = oracle.Oracle.for_stream(s, stream_release=stream_release)
    mixed = oracle.Oracle.for_stream(s, stream_release=stream_release)
    mixed.push_batch(_empty(s))
    assert len(mixed.drain().records) == 0
    for b in range(s.n_batches):
        bt = s.batch(b)
        plain.push_batch(bt)
        mixed.push_batch(bt)
        mixed.push_batch(_empty(s))
        want, got = plain.drain(), mixed.drain()
        assert got.status == want.status == 0
        assert np.array_equal(got.records.view(np.uint8), want.records.view(np.uint8)), b
        assert np.array_equal(got.payload, want.payload), b
        assert np.array_equal(got.topk.view(np.uint8), want.topk.view(np.uint8)), b
        mixed.push_batch(_empty(s))
        assert len(mixed.drain().records) == 0
    plain.close()
    mixed.close()
