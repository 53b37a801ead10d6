"""CUDA path vs the oracle, bit for bit, through the C ABI."""
import json
import os
import random

import numpy as np
import pytest

torch = pytest.importorskip("torch")

import paper_2403_04311_gb300 as alto
from fragments import split, to_batch, tree_fragments
from gen import make_stream
from gpu_harness import (assert_same, gpu_drain_host, run_both_stream, run_gpu_batches, run_oracle_batches,
                         small_caps, stream_caps)

pytestmark = pytest.mark.gpu
GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


@pytest.mark.parametrize("name", ["tiny", "tiny64", "factcheck", "throughput", "tokens", "adversarial", "tot"])
@pytest.mark.parametrize("drain_every", [1, 3])
@pytest.mark.parametrize("launch", ["graph", "direct"])
def test_workloads_small(name, drain_every, launch):
    """Pushes of these small streams replay the captured push graph by
    default; with ALTO_FLAG_DIRECT_LAUNCH every kernel is launched by itself."""
    s = make_stream(name, small=True)
    caps = dict(stream_caps(s), direct_launch=(launch == "direct"))
    o, g = run_both_stream(s, drain_every=drain_every, caps=caps)
    assert all(d.status == 0 for d in o)
    assert_same(o, g, f"{name}/{drain_every}/{launch}")


@pytest.mark.parametrize("mode", ["stages", "hot"])
def test_graph_replays_while_profiling(mode):
    """With profiling on, a replayed push records its stage-boundary events
    through the graph's event-record nodes (fresh events every push): the
    records still match the oracle and the timed stages have device time."""
    s = make_stream("factcheck", small=True)
    agg = alto.Aggregator(s.depth, s.payload_op, s.score_op, s.topk_k, **stream_caps(s))
    agg.profile(alto.PROFILE_STAGES if mode == "stages" else alto.PROFILE_HOT)
    import oracle
    o = oracle.Oracle.for_stream(s)
    for b in range(s.n_batches):
        bt = s.batch(b)
        db = alto.to_device(bt)
        assert agg.push(db.tags, db.off, db.payload, db.score) == alto.OK
        o.push_batch(bt)
        assert_same([o.drain()], [gpu_drain_host(agg.drain())], f"{mode} batch {b}")
    st, prof = agg.profile_read()
    agg.profile(False)
    agg.close()
    o.close()
    assert st == alto.OK and prof["pushes"] == s.n_batches
    assert prof["stage_ms"]["gather"] > 0.0
    if mode == "stages":
        assert prof["stage_ms"]["ingest"] > 0.0 and prof["stage_ms"]["records"] > 0.0


def test_golden_factool_claims():
    fx = json.load(open(os.path.join(GOLDEN, "factool_claims.json")))
    frags = [(tuple(tuple(t) for t in f["tags"]), f["tokens"], f["score"]) for f in fx["fragments"]]
    batches = [to_batch(p, fx["depth"], True) for p in split(frags, fx["batches"])]
    _, g = run_gpu_batches(fx["depth"], fx["payload_op"], fx["score_op"], fx["topk_k"], batches,
                           small_caps(8, 16, fx["depth"]))
    o = run_oracle_batches(fx["depth"], fx["payload_op"], fx["score_op"], fx["topk_k"], batches)
    assert_same(o, g, "golden")
    _st, rec, pay, tk = g[1]
    assert pay.tolist() == fx["drains"][1]["payload"]
    assert rec["parent_id"].tolist() == [41, 40, 7]


def test_golden_errors_detected_on_device():
    fx = json.load(open(os.path.join(GOLDEN, "errors.json")))
    for case in fx["cases"]:
        if "closed" in case["name"]:
            continue  # a repeat across batches of an emitted group: not in the device scope
        frags = [(tuple(tuple(t) for t in f["tags"]), f["tokens"], 0.0) for f in case["fragments"]]
        batches = []
        for part in split(frags, case["batches"]):
            b = to_batch(part, fx["depth"], False)
            if case.get("bad_offsets"):
                b["off"][1], b["off"][2] = b["off"][2], b["off"][1]
            batches.append(b)
        _, g = run_gpu_batches(fx["depth"], fx["payload_op"], fx["score_op"], fx["topk_k"], batches,
                               small_caps(8, 16, fx["depth"]))
        assert [d[0] for d in g] == case["status"], case["name"]


def _brute_cases(seed=0, count=150):
    rng = random.Random(seed)
    shapes = [3, [2, 1], [1, 3, 2], [[2, 1], [3]], [[1], [2, 2], [1]], [[2, [1, 2]], [1, [1]]][:0]]
    shapes = [3, [2, 1], [1, 3, 2], [[2, 1], [3]], [[1], [2, 2], [1]], [[[1, 2], [1]], [[2]]]]
    out = []
    for _ in range(count):
        shape = rng.choice(shapes)
        depth = 1
        x = shape
        while not isinstance(x, int):
            x = x[0]
            depth += 1
        frags = tree_fragments(shape, score_fn=lambda k: [-1.0, -0.0, 0.0, 0.5, 0.5, 2.0, -3.5][k % 7])
        rng.shuffle(frags)
        n = len(frags)
        cuts, left = [], n
        while left:
            c = rng.randint(1, left)
            cuts.append(c)
            left -= c
        po = [0] * depth
        if rng.random() < 0.8:
            po[depth - 1] = 1
        so = [rng.choice([0, 1, 2]) for _ in range(depth)]
        kk = [rng.choice([1, 2, 3]) if x == 2 else 0 for x in so]
        out.append((depth, po, so, kk, frags, cuts))
    return out


def test_bruteforce_streams_on_device():
    for depth, po, so, kk, frags, cuts in _brute_cases():
        ws = any(x != 0 for x in so)
        batches = [to_batch(p, depth, ws) for p in split(frags, cuts)]
        _, g = run_gpu_batches(depth, po, so, kk, batches, small_caps(len(frags), 64, depth))
        o = run_oracle_batches(depth, po, so, kk, batches)
        assert_same(o, g, f"{depth} {po} {so} {kk} {cuts}")


def test_bruteforce_streams_on_device_direct_launch():
    """A share of the brute-force streams with every kernel launched by itself."""
    for depth, po, so, kk, frags, cuts in _brute_cases()[::3]:
        ws = any(x != 0 for x in so)
        batches = [to_batch(p, depth, ws) for p in split(frags, cuts)]
        caps = dict(small_caps(len(frags), 64, depth), direct_launch=True)
        _, g = run_gpu_batches(depth, po, so, kk, batches, caps)
        o = run_oracle_batches(depth, po, so, kk, batches)
        assert_same(o, g, f"direct {depth} {po} {so} {kk} {cuts}")


def test_leaf_slot_repeated_in_a_later_batch():
    """A leaf slot below 256 given again in a later batch while its group is
    still open: the oracle and the device both report EDUP in that batch."""
    for c in (0, 5, 255):
        frags = [(((9, 0, 1), (90, c, 0)), [1], 0.0),
                 (((9, 0, 1), (90, c, 0)), [2], 0.0),
                 (((9, 0, 1), (90, c + 1, 1)), [3], 0.0)]
        batches = [to_batch(p, 2, False) for p in split(frags, [1, 2])]
        o = run_oracle_batches(2, [0, 1], [0, 0], [0, 0], batches)
        _, g = run_gpu_batches(2, [0, 1], [0, 0], [0, 0], batches, small_caps(4, 16, 2))
        assert [d.status for d in o] == [alto.OK, alto.EDUP]
        assert [d[0] for d in g] == [alto.OK, alto.EDUP], c


def test_nan_score_is_einval():
    frags = tree_fragments([2], score_fn=lambda k: float("nan") if k == 1 else 1.0)
    b = to_batch(frags, 2, True)
    _, g = run_gpu_batches(2, [0, 1], [0, 1], [0, 0], [b], small_caps(4, 16, 2))
    assert g[0][0] == alto.EINVAL


def test_poisoned_handle_and_destroy():
    frags = tree_fragments([2, 2])
    bad = list(frags) + [frags[0]]     # duplicate leaf in the batch
    agg = alto.Aggregator(2, [0, 1], [0, 0], None, **small_caps(8, 64, 2))
    db = alto.to_device(to_batch(bad, 2, False))
    assert agg.push(db.tags, db.off, db.payload) == alto.OK     # device error: found later
    assert agg.drain().status == alto.EDUP
    db2 = alto.to_device(to_batch(frags, 2, False))
    assert agg.push(db2.tags, db2.off, db2.payload) == alto.EDUP
    assert agg.drain().status == alto.EDUP
    agg.close()


def test_output_capacity_is_enospc():
    s = make_stream("tiny64")
    caps = stream_caps(s)
    caps["out_records"] = 5
    _, g = run_gpu_batches(s.depth, s.payload_op, s.score_op, s.topk_k, [s.batch(0)], caps)
    assert g[0][0] == alto.ENOSPC


@pytest.mark.parametrize("leaf", ["accumulate", "topk", "stream_release"])
def test_full_open_group_table_is_enospc(leaf):
    """2,001 open groups in one batch and a table of 1,024 slots: the inserts
    that find no slot end the batch with ENOSPC, and no other class (the
    unplaced groups must not be taken for one another, which would read as
    repeated leaf slots), on each leaf form."""
    frags = tree_fragments([2] * 2000)
    n_pay = sum(len(f[1]) for f in frags)
    topk = leaf == "topk"
    caps = small_caps(len(frags), n_pay, 2)
    caps.update(max_open_groups=16, stream_release=(leaf == "stream_release"))
    agg = alto.Aggregator(2, [0, 1], [0, 2 if topk else 0], [0, 2 if topk else 0], **caps)
    db = alto.to_device(to_batch(frags, 2, topk))
    assert agg.push(db.tags, db.off, db.payload, db.score if topk else None) == alto.OK
    d = agg.drain()
    assert d.status == alto.ENOSPC
    assert agg.drain().status == alto.ENOSPC      # latched
    agg.close()


def test_host_argument_errors_do_not_poison():
    frags = tree_fragments([2, 1])
    agg = alto.Aggregator(2, [0, 1], [0, 0], None, **small_caps(4, 16, 2))
    db = alto.to_device(to_batch(frags, 2, False))
    big = alto.to_device(to_batch(frags + tree_fragments([3], id_base=900), 2, False))
    assert agg.push(big.tags, big.off, big.payload) == alto.EINVAL   # n above max_batch_fragments
    assert agg.push(db.tags, db.off, db.payload) == alto.OK
    d = agg.drain()
    assert d.status == alto.OK
    rec, pay, _ = d.host()
    assert len(rec) == 3
    agg.close()


def test_determinism_repeated_runs():
    s = make_stream("adversarial", small=True)
    _, g1 = run_both_stream(s, drain_every=2)
    _, g2 = run_both_stream(s, drain_every=2)
    for a, b in zip(g1, g2):
        assert a[0] == b[0]
        assert np.array_equal(a[1].view(np.uint8), b[1].view(np.uint8))
        assert np.array_equal(a[2], b[2])


def _wide_topk_stream(n_children, leaves_per_child, batches, seed):
    """Depth 2: one source whose level-0 group has n_children child groups
    (TOPK(5) over them, CONCAT inside each), all in a shuffled order."""
    rng = np.random.default_rng(seed)
    frags = []
    for c in range(n_children):
        for k in range(leaves_per_child):
            tags = ((1, c, c == n_children - 1), (100 + c, k, k == leaves_per_child - 1))
            frags.append((tags, rng.integers(0, 1000, size=int(rng.integers(1, 6))).tolist(),
                          float(rng.standard_normal())))
    order = rng.permutation(len(frags))
    frags = [frags[i] for i in order]
    cuts = np.linspace(0, len(frags), batches + 1).astype(int)
    return [frags[a:b] for a, b in zip(cuts[:-1], cuts[1:])]


@pytest.mark.parametrize("n_children,batches", [(10_000, 1), (12_000, 3)])
def test_topk_level_with_a_segment_longer_than_a_warp_share(n_children, batches):
    """An upper TOPK level whose group has more than 4,096 items in one batch
    takes the block-wide reduce; bit for bit against the oracle."""
    parts = _wide_topk_stream(n_children, 2, batches, seed=n_children)
    bts = [to_batch(p, 2, True) for p in parts]
    n = max(b["n"] for b in bts)
    pay = max(len(b["payload"]) for b in bts)
    caps = dict(max_batch_fragments=n, max_batch_payload=pay, max_open_groups=1 << 16, arena_elems=1 << 22,
                out_records=n_children + 64, out_payload_elems=sum(len(b["payload"]) for b in bts) + 64,
                out_topk=64, max_emit_children=2 * n_children * 2 + 64)
    po, so, kk = [0, 1], [2, 1], [5, 0]
    _, g = run_gpu_batches(2, po, so, kk, bts, caps)
    o = run_oracle_batches(2, po, so, kk, bts)
    assert all(d.status == 0 for d in o)
    assert_same(o, g, f"wide topk {n_children}/{batches}")
