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
from gpu_harness import route_release_and_aggregate, route_stream_vs_oracle

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("name,level", [("factcheck", 1), ("throughput", 1), ("tot", 0), ("adversarial", 2)])
@pytest.mark.parametrize("R", [1, 3, 8])
@pytest.mark.parametrize("policy", [alto.ROUTE_HASH, alto.ROUTE_LEAST_LOADED])
def test_route_matches_oracle(name, level, R, policy):
    route_stream_vs_oracle(make_stream(name, small=True), level, R, policy)


def test_route_many_replicas():
    route_stream_vs_oracle(make_stream("throughput", small=True), 2, 1000, alto.ROUTE_LEAST_LOADED)
    route_stream_vs_oracle(make_stream("throughput", small=True), 2, 1000, alto.ROUTE_HASH)


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
    route_stream_vs_oracle(make_stream("throughput"), 1, 8, alto.ROUTE_LEAST_LOADED, batches=range(4))
