"""Edge cases of the CUDA path against the oracle, bit for bit, through the C
ABI: a small open-group table and a small flow table whose deleted slots
must be taken again, empty batches, the largest depth, parent ids and k, two
output rings, and batches around a warp and a sort/scan tile.  (This file
runs after the main parity files.)"""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

from fragments import split, to_batch, tree_fragments, window_stream
from gen import make_stream
from gpu_harness import (assert_same, route_release_and_aggregate, route_stream_vs_oracle, run_both_stream,
                         run_gpu_batches, run_oracle_batches, small_caps, stream_caps)

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("leaf", ["accumulate", "topk", "stream_release"])
def test_small_table_reuses_deleted_slots(leaf):
    """20,000 groups through a 1,024-slot table, never more than 200 of them
    open at once (80,000 leaves in 256-fragment batches): inserts must take
    the slots of emitted groups.  Without that, slots left deleted behind
    live keys fill the table within about fifty batches (ENOSPC); with it,
    every drain matches the oracle bit for bit."""
    s = window_stream(20_000, 4, 200, 256, seed=7, topk=(leaf == "topk"))
    caps = stream_caps(s)
    caps["max_open_groups"] = 256                 # 1,024 slots
    o, g = run_both_stream(s, drain_every=1, caps=caps, stream_release=(leaf == "stream_release"))
    assert all(d.status == 0 for d in o)
    assert_same(o, g, f"window/{leaf}")


def _empty_batch(s):
    return dict(n=0, seq_base=0, tags=np.zeros((s.depth, 0), np.uint64), off=np.zeros(1, np.uint32),
                payload=np.zeros(0, np.int32), score=None if s.score is None else np.zeros(0, np.float32))


@pytest.mark.parametrize("name,stream_release", [("factcheck", False), ("throughput", False),
                                                 ("throughput", True)])
def test_empty_batches_are_no_ops(name, stream_release):
    """An empty batch before, between and after the stream's batches, and a
    drain after nothing but empty pushes: every drain equals the oracle's,
    which is given the same empty batches (no group changes, nothing is
    emitted or released)."""
    s = make_stream(name, small=True)
    batches = [_empty_batch(s), _empty_batch(s)]
    for b in range(s.n_batches):
        batches += [s.batch(b), _empty_batch(s)]
    caps = stream_caps(s, stream_release=stream_release)
    if stream_release:
        caps["stream_release"] = True
    _, g = run_gpu_batches(s.depth, s.payload_op, s.score_op, s.topk_k, batches, caps)
    o = run_oracle_batches(s.depth, s.payload_op, s.score_op, s.topk_k, batches, stream_release=stream_release)
    assert all(d.status == 0 for d in o)
    assert_same(o, g, f"{name} with empty batches")
    assert len(g[0][1]) == 0 and len(g[1][1]) == 0


def _deep_forest(seed, n_roots=4, depth=8):
    """Random trees of the largest depth, fanout 1-2 per level and 1-40
    leaves per leaf parent, with each level's parent ids remapped to the
    top of the u32 range (the first group met at a level gets 0xFFFFFFFF)."""
    rng = np.random.default_rng(seed)

    def shape(d):
        if d == 1:
            return int(rng.integers(1, 41))
        return [shape(d - 1) for _ in range(int(rng.integers(1, 3)))]

    frags = []
    for r in range(n_roots):
        frags += tree_fragments(shape(depth), id_base=100_000 * (r + 1),
                                score_fn=lambda k: float(rng.standard_normal()),
                                tok_fn=lambda k: [int(x) for x in rng.integers(0, 50257, int(rng.integers(0, 5)))])
    remap = [{} for _ in range(depth)]
    out = []
    for tags, tok, sc in frags:
        nt = []
        for l, (p_, c, last) in enumerate(tags):
            m = remap[l].setdefault(p_, 0xFFFFFFFF - len(remap[l]))
            nt.append((m, c, last))
        out.append((tuple(nt), tok, sc))
    order = rng.permutation(len(out))
    out = [out[i] for i in order]
    cuts = sorted(rng.choice(np.arange(1, len(out)), size=4, replace=False).tolist())
    sizes = [b - a for a, b in zip([0] + cuts, cuts + [len(out)])]
    return out, sizes


@pytest.mark.parametrize("ops", [
    # CONCAT at the leaf parent, TOPK(32) over its level's groups, MAX above
    dict(payload_op=[0, 0, 0, 0, 0, 0, 0, 1], score_op=[0, 0, 1, 0, 0, 0, 2, 0],
         topk_k=[0, 0, 0, 0, 0, 0, 32, 0]),
    # CONCAT four levels above the leaf parent, TOPK(32) over leaves, MAX at the root
    dict(payload_op=[0, 0, 0, 1, 0, 0, 0, 0], score_op=[1, 0, 0, 0, 0, 0, 0, 2],
         topk_k=[0, 0, 0, 0, 0, 0, 0, 32]),
])
@pytest.mark.parametrize("seed", [1, 2])
def test_depth8_top_ids_and_k32(ops, seed):
    """The largest depth (8 tags), parent ids at the top of the u32 range
    (0xFFFFFFFF included) and the largest k (32, above and below the child
    counts), in five batches of a random arrival order, bit for bit against
    the oracle."""
    D = 8
    frags, sizes = _deep_forest(seed, depth=D)
    batches = [to_batch(part, D, True) for part in split(frags, sizes)]
    n_pay = max(int(b["off"][-1]) for b in batches)
    caps = small_caps(max(sizes), n_pay, D)
    caps.update(arena_elems=1 << 22, out_records=1 << 14, out_payload_elems=1 << 16, out_topk=1 << 16,
                max_emit_children=1 << 14)
    _, g = run_gpu_batches(D, ops["payload_op"], ops["score_op"], ops["topk_k"], batches, caps)
    o = run_oracle_batches(D, ops["payload_op"], ops["score_op"], ops["topk_k"], batches)
    assert all(d.status == 0 for d in o)
    assert sum(len(d.records) for d in o) > 100
    assert_same(o, g, f"depth 8 seed {seed}")


def test_route_small_flow_table_reuses_released_slots():
    """20,000 flows, at most 200 live at once, through a flow table of 1,024
    slots, routed into four GPU aggregators and released from their records:
    new flows must take the slots of released ones."""
    route_release_and_aggregate(window_stream(20_000, 4, 200, 256, seed=7), max_flows=256)


@pytest.mark.parametrize("name,stream_release", [("factcheck", False), ("throughput", True)])
def test_double_ring_keeps_a_drain_through_the_next(name, stream_release):
    """With two output rings, what a drain returns stays intact through the
    next push and drain: each drain's records, payload and top-k pairs, read
    back only after the following push and drain, equal the oracle's."""
    import oracle
    import paper_2403_04311_gb300 as alto

    s = make_stream(name, small=True)
    caps = stream_caps(s, stream_release=stream_release)
    caps.update(double_ring=True, stream_release=stream_release)
    agg = alto.Aggregator(s.depth, s.payload_op, s.score_op, s.topk_k, **caps)
    o = oracle.Oracle.for_stream(s, stream_release=stream_release)

    def check(pending, b):
        d, od = pending
        rec, pay, tk = d.host()
        assert np.array_equal(rec.view(np.uint8), od.records.view(np.uint8)), b
        assert np.array_equal(pay, od.payload), b
        assert np.array_equal(tk.view(np.uint8), od.topk.view(np.uint8)), b

    pending, n_rec = None, 0
    for b in range(s.n_batches):
        bt = s.batch(b)
        db = alto.to_device(bt)
        assert agg.push(db.tags, db.off, db.payload, db.score) == alto.OK
        d = agg.drain()
        assert d.status == alto.OK
        o.push_batch(bt)
        od = o.drain()
        n_rec += len(od.records)
        if pending is not None:
            check(pending, b - 1)
        pending = (d, od)
    check(pending, s.n_batches - 1)
    agg.close()
    o.close()
    assert s.n_batches > 2 and n_rec > 0


_BOUNDARY_SIZES = [1, 31, 32, 33, 4095, 4096, 4097, 8191, 8192, 8193]


def _boundary_batches(s):
    """The stream cut into batches of 1, 31, 32, 33, 4,095, 4,096, 4,097,
    8,191, 8,192 and 8,193 fragments and the rest: around a warp (32), the
    tile of the radix sort and the scans (4,096 elements), and the largest
    sort one CTA takes in shared memory (8,192 pairs; graph replays of pushes
    up to 8K fragments launch only that form, larger ones both)."""
    import dataclasses

    sizes = _BOUNDARY_SIZES + [s.n - sum(_BOUNDARY_SIZES)]
    assert sizes[-1] > 0
    return dataclasses.replace(s, batch_sizes=np.asarray(sizes))


@pytest.mark.parametrize("leaf", ["accumulate", "topk", "stream_release"])
def test_batches_at_warp_and_tile_boundaries(leaf):
    """Every leaf form on batches around a warp and a sort/scan tile, bit for
    bit against the oracle."""
    s = _boundary_batches(window_stream(40_000, 4, 200, 256, seed=11, topk=(leaf == "topk")))
    o, g = run_both_stream(s, drain_every=1, stream_release=(leaf == "stream_release"))
    assert all(d.status == 0 for d in o)
    assert_same(o, g, f"boundary batches/{leaf}")


@pytest.mark.parametrize("policy", ["hash", "least_loaded"])
@pytest.mark.parametrize("R", [8, 1000])
def test_route_batches_at_warp_and_tile_boundaries(policy, R):
    """Routing on batches around a warp and a sort/scan tile: each batch's
    replicas, stable partition (one radix pass for 8 replicas, two for 1,000)
    and sub-batches equal the routing oracle's."""
    import paper_2403_04311_gb300 as alto

    s = _boundary_batches(window_stream(40_000, 4, 200, 256, seed=11))
    route_stream_vs_oracle(s, 1, R, alto.ROUTE_HASH if policy == "hash" else alto.ROUTE_LEAST_LOADED)
