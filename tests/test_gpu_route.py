"""Routing on the GPU against the routing oracle, bit for bit, through the C ABI.

Per batch: each fragment's replica, the stable partition (perm), the replica
offsets, and every replica's sub-batch (tags, payload offsets, payload,
scores).  Flows placed by load persist across batches and are released by
the aggregators' records; the end-to-end test routes a stream into GPU
aggregators and checks every group at or below the routing level against a
single oracle aggregator (Sec. 4.3).
"""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

import oracle
import paper_2403_04311_gb300 as alto
from gen import make_stream
from gpu_harness import route_release_and_aggregate

pytestmark = pytest.mark.gpu


def _route_stream(s, level, R, policy, batches=None, max_flows=0):
    bsz = int(max(s.batch_sizes))
    pay = max(int(s.off[st1] - s.off[st0]) for st0, st1 in zip(s.batch_starts()[:-1], s.batch_starts()[1:]))
    rt = alto.Router(s.depth, level, R, policy, max_batch_fragments=bsz, max_batch_payload=max(pay, 1),
                     max_flows=max_flows, with_score=s.score is not None)
    ro = oracle.RouterOracle(s.depth, level, R, policy)
    for b in (range(s.n_batches) if batches is None else batches):
        bt = s.batch(b)
        db = alto.to_device(bt)
        assert rt.route(db.tags, db.off, db.payload, db.score) == alto.OK
        st, fo, po = rt.counts()
        assert st == alto.OK
        replica, perm, counts, parts = ro.route(bt)
        assert np.array_equal(fo, counts)
        rep_d, perm_d, parts_d = rt.outputs(fo, po)
        assert np.array_equal(rep_d.cpu().numpy(), replica)
        assert np.array_equal(perm_d.cpu().numpy(), perm)
        for r in range(R):
            t, o, p, sc = parts_d[r]
            want = parts[r]
            assert np.array_equal(t.cpu().numpy().view(np.uint64), want["tags"]), (b, r)
            assert np.array_equal(o.cpu().numpy().astype(np.int64), want["off"]), (b, r)
            assert np.array_equal(p.cpu().numpy(), want["payload"]), (b, r)
            if want["score"] is not None:
                assert np.array_equal(sc.cpu().numpy().view(np.uint32), want["score"].view(np.uint32))
    rt.close()


@pytest.mark.parametrize("name,level", [("factcheck", 1), ("throughput", 1), ("tot", 0), ("adversarial", 2)])
@pytest.mark.parametrize("R", [1, 3, 8])
@pytest.mark.parametrize("policy", [alto.ROUTE_HASH, alto.ROUTE_LEAST_LOADED])
def test_route_matches_oracle(name, level, R, policy):
    _route_stream(make_stream(name, small=True), level, R, policy)


def test_route_many_replicas():
    _route_stream(make_stream("throughput", small=True), 2, 1000, alto.ROUTE_LEAST_LOADED)
    _route_stream(make_stream("throughput", small=True), 2, 1000, alto.ROUTE_HASH)


def test_route_errors():
    n = 3000       # 3,000 flows for a table of 1,024 slots
    tags = np.zeros((2, n), dtype=np.uint64)
    tags[0] = (np.uint64(1) << np.uint64(32)) | np.arange(n, dtype=np.uint64)
    tags[1] = ((np.arange(n, dtype=np.uint64) + np.uint64(1000)) << np.uint64(32)) | (np.uint64(1) << np.uint64(31))
    bt = dict(n=n, tags=tags, off=np.arange(n + 1, dtype=np.uint32), payload=np.arange(n, dtype=np.int32),
              score=None)
    rt = alto.Router(2, 1, 4, alto.ROUTE_LEAST_LOADED, max_batch_fragments=n, max_batch_payload=n, max_flows=4)
    db = alto.to_device(bt)
    assert rt.route(db.tags, db.off, db.payload) == alto.OK
    st, _, _ = rt.counts()
    assert st == alto.ENOSPC
    assert rt.route(db.tags, db.off, db.payload) == alto.ENOSPC       # latched
    rt.close()
    bad = dict(bt)
    bad["off"] = bt["off"].copy()
    bad["off"][1], bad["off"][2] = bad["off"][2], bad["off"][1]
    rt = alto.Router(2, 1, 4, alto.ROUTE_HASH, max_batch_fragments=n, max_batch_payload=n)
    db = alto.to_device(bad)
    assert rt.route(db.tags, db.off, db.payload) == alto.OK
    st, _, _ = rt.counts()
    assert st == alto.EINVAL
    rt.close()


def test_route_release_and_aggregate():
    """Route at level 1 into R GPU aggregators, release completed flows from
    their device records, and compare with the oracle router + one oracle
    aggregator: replicas match batch by batch, and every group at level >= 1
    gets the record the whole stream gives."""
    route_release_and_aggregate(make_stream("factcheck", small=True))


@pytest.mark.slow
def test_route_fullsize_throughput():
    """The 16M-fragment throughput stream, 1M batches, eight replicas placed by load."""
    _route_stream(make_stream("throughput"), 1, 8, alto.ROUTE_LEAST_LOADED, batches=range(4))
