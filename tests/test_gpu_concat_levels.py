"""CONCAT at a level M above the leaf parent (M < D-1): CUDA path vs the oracle,
bit for bit, through the C ABI.

A group of a level between M and the leaf parent completes into one span of
its parent's arena vectors; the level-M group then concatenates its children's
spans in child-index order (Sec. 3.2: the outputs of the nested pmaps are put
back into stream order at the aggregation point).  The cases cover the atomic
(no TOPK) and the sorted (TOPK) level paths, groups spanning many batches,
several scan tiles of dense slots, and the one-shot entry point.
"""
import dataclasses
import json
import os
import random

import pytest

torch = pytest.importorskip("torch")

import paper_2403_04311_gb300 as alto
from fragments import split, to_batch, tree_fragments
from gen import make_stream
from gpu_harness import assert_same, run_both_stream, run_gpu_batches, run_oracle_batches, stream_caps

pytestmark = pytest.mark.gpu
GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def small_caps(n, payload):
    return dict(max_batch_fragments=max(n, 1), max_batch_payload=max(payload, 1),
                max_open_groups=4096, arena_elems=1 << 16, out_records=4096,
                out_payload_elems=1 << 14, out_topk=4096, max_emit_children=4096)


def chain_caps(s):
    """Capacities for a stream whose CONCAT level sits above the leaf parent:
    children of every level may take dense slots in one batch, and a leaf's
    tokens may sit in two levels' vectors at once while they are handed up."""
    caps = stream_caps(s, arena_factor=6)
    caps["max_emit_children"] = s.n * s.depth + 16
    return caps


def with_concat_at(s, m):
    po = [0] * s.depth
    po[m] = 1
    return dataclasses.replace(s, payload_op=tuple(po))


def test_golden_docs_concat_claim():
    fx = json.load(open(os.path.join(GOLDEN, "factool_docs_concat_claim.json")))
    frags = [(tuple(tuple(t) for t in f["tags"]), f["tokens"], f["score"]) for f in fx["fragments"]]
    batches = [to_batch(p, fx["depth"], False) for p in split(frags, fx["batches"])]
    _, g = run_gpu_batches(fx["depth"], fx["payload_op"], fx["score_op"], fx["topk_k"], batches,
                           small_caps(8, 32))
    o = run_oracle_batches(fx["depth"], fx["payload_op"], fx["score_op"], fx["topk_k"], batches)
    assert_same(o, g, "golden")
    for k, want in enumerate(fx["drains"]):
        st, rec, pay, _ = g[k]
        assert st == want["status"]
        assert pay.tolist() == want["payload"]
        assert rec["payload_len"].tolist() == [r["payload_len"] for r in want["records"]]


def _chain_cases(seed, count):
    rng = random.Random(seed)
    shapes = [[2, 1], [1, 3, 2], [[2, 1], [3]], [[1], [2, 2], [1]], [[[1, 2], [1]], [[2]]],
              [[[3], [1, 1]], [[2, 2]], [[1]]], [[[[2], [1]], [[1, 1]]], [[[3]]]]]
    out = []
    for _ in range(count):
        shape = rng.choice(shapes)
        depth = 1
        x = shape
        while not isinstance(x, int):
            x = x[0]
            depth += 1
        frags = tree_fragments(shape, score_fn=lambda k: [-1.0, -0.0, 0.0, 0.5, 0.5, 2.0, -3.5][k % 7],
                               tok_fn=lambda k: list(range(1000 * k, 1000 * k + (k % 4))))
        rng.shuffle(frags)
        n = len(frags)
        cuts, left = [], n
        while left:
            c = rng.randint(1, left)
            cuts.append(c)
            left -= c
        po = [0] * depth
        po[rng.randrange(0, depth - 1)] = 1
        so = [rng.choice([0, 1, 2]) for _ in range(depth)]
        kk = [rng.choice([1, 2, 3]) if x == 2 else 0 for x in so]
        out.append((depth, po, so, kk, frags, cuts))
    return out


def test_bruteforce_concat_above_leaf_parent():
    for depth, po, so, kk, frags, cuts in _chain_cases(seed=11, count=200):
        ws = any(x != 0 for x in so)
        batches = [to_batch(p, depth, ws) for p in split(frags, cuts)]
        _, g = run_gpu_batches(depth, po, so, kk, batches, small_caps(len(frags), 256))
        o = run_oracle_batches(depth, po, so, kk, batches)
        assert_same(o, g, f"{depth} {po} {so} {kk} {cuts}")


@pytest.mark.parametrize("name,m", [("throughput", 0), ("throughput", 1), ("throughput", 2),
                                    ("factcheck", 1), ("factcheck", 2),
                                    ("adversarial", 2), ("adversarial", 4)])
@pytest.mark.parametrize("drain_every", [1, 3])
def test_workloads_concat_moved_up(name, m, drain_every):
    s = with_concat_at(make_stream(name, small=True), m)
    o, g = run_both_stream(s, drain_every=drain_every, caps=chain_caps(s))
    assert all(d.status == 0 for d in o)
    assert_same(o, g, f"{name} M={m}/{drain_every}")


def test_arena_returns_to_empty():
    """Every group completes by the end of the stream: all chunks of every
    level's vectors are back on the free stacks."""
    s = with_concat_at(make_stream("throughput", small=True), 1)
    agg = alto.Aggregator(s.depth, s.payload_op, s.score_op, s.topk_k, **chain_caps(s))
    for b in range(s.n_batches):
        db = alto.to_device(s.batch(b))
        assert agg.push(db.tags, db.off, db.payload, db.score) == alto.OK
        if b % 4 == 3:
            assert agg.drain().status == alto.OK
    assert agg.drain().status == alto.OK
    st, open_groups, arena_used = agg.stats()
    agg.close()
    assert st == alto.OK
    assert open_groups == 0
    assert arena_used == 0
