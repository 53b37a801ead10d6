"""The routing oracle against facts it does not compute itself.

* splitmix64: the generator's published first output for seed 0
  (0x9E3779B97F4A7C15 mixed = 0xE220A8397B1DCDAF);
* invariants: one replica per flow (within a batch and, for LEAST_LOADED,
  across batches until released); the partition is a permutation, stable
  (arrival order kept inside a replica), and each sub-batch carries exactly
  its fragments' tags, payload and scores;
* LEAST_LOADED with equal loads gives the first R new flows R different
  replicas, and flows go to the replica that has routed the fewest fragments;
* release: a flow reported complete is placed afresh;
* Sec. 4.3, end to end: routing the stream at level L and aggregating every
  replica's sub-batches separately gives, for every group at a level >= L,
  the record the whole stream gives on one aggregator (records at levels < L
  span replicas and are not compared).
"""
import numpy as np

import oracle
from gen import make_stream


def test_splitmix64_published_vector():
    assert oracle.splitmix64_mix(0x9E3779B97F4A7C15) == 0xE220A8397B1DCDAF


def _check_partition(batch, replica, perm, counts, parts, R):
    n = batch["n"]
    assert sorted(perm.tolist()) == list(range(n))
    assert counts[0] == 0 and counts[-1] == n
    for r in range(R):
        idx = perm[counts[r]:counts[r + 1]]
        assert np.all(replica[idx] == r)
        assert np.all(np.diff(idx) > 0)                  # stable
        p = parts[r]
        assert p["n"] == len(idx)
        assert np.array_equal(p["tags"], batch["tags"][:, idx])
        want = [batch["payload"][batch["off"][i]:batch["off"][i + 1]] for i in idx]
        got = [p["payload"][p["off"][k]:p["off"][k + 1]] for k in range(len(idx))]
        assert all(np.array_equal(a, b) for a, b in zip(want, got))
        if batch["score"] is not None:
            assert np.array_equal(p["score"], batch["score"][idx])


def test_partition_and_flow_invariants():
    s = make_stream("factcheck", small=True)
    for policy in (oracle.HASH, oracle.LEAST_LOADED):
        for R in (1, 3, 8):
            ro = oracle.RouterOracle(s.depth, 1, R, policy)
            seen = {}
            for b in range(s.n_batches):
                bt = s.batch(b)
                replica, perm, counts, parts = ro.route(bt)
                _check_partition(bt, replica, perm, counts, parts, R)
                pids = (bt["tags"][1] >> np.uint64(32)).tolist()
                for p, r in zip(pids, replica.tolist()):
                    assert seen.setdefault(p, r) == r


def test_least_loaded_spreads_new_flows():
    def frag(pid, c):
        return (np.uint64(pid) << np.uint64(32)) | np.uint64(c)
    # one batch, 5 new flows, R = 5: all different replicas
    tags = np.asarray([[frag(1, 0)] * 5, [frag(100 + k, 0) for k in range(5)]], dtype=np.uint64)
    bt = dict(n=5, tags=tags, off=np.arange(6), payload=np.arange(5, dtype=np.int32), score=None)
    ro = oracle.RouterOracle(2, 1, 5, oracle.LEAST_LOADED)
    replica, _, _, _ = ro.route(bt)
    assert sorted(replica.tolist()) == [0, 1, 2, 3, 4]
    # flow 100 keeps its replica and adds 3 fragments to its load; in the next
    # batch (loads are taken at the batch start) a new flow avoids that replica
    tags2 = np.asarray([[frag(1, 0)] * 3, [frag(100, 1), frag(100, 2), frag(100, 3)]], dtype=np.uint64)
    bt2 = dict(n=3, tags=tags2, off=np.arange(4), payload=np.arange(3, dtype=np.int32), score=None)
    replica2, _, _, _ = ro.route(bt2)
    r100 = replica[0]
    assert replica2.tolist() == [r100] * 3
    tags3 = np.asarray([[frag(1, 0)], [frag(200, 0)]], dtype=np.uint64)
    bt3 = dict(n=1, tags=tags3, off=np.arange(2), payload=np.arange(1, dtype=np.int32), score=None)
    replica3, _, _, _ = ro.route(bt3)
    assert replica3[0] == min(r for r in range(5) if r != r100)


def test_release_places_a_flow_afresh():
    def frag(pid):
        return np.uint64(pid) << np.uint64(32)
    ro = oracle.RouterOracle(2, 1, 2, oracle.LEAST_LOADED)
    mk = lambda pids: dict(n=len(pids), tags=np.asarray([[frag(1)] * len(pids), [frag(p) for p in pids]],
                                                          dtype=np.uint64),
                           off=np.arange(len(pids) + 1), payload=np.arange(len(pids), dtype=np.int32), score=None)
    r1, _, _, _ = ro.route(mk([7, 7, 7]))          # flow 7 -> replica 0, load 3
    r2, _, _, _ = ro.route(mk([8]))                # flow 8 -> replica 1
    assert r1.tolist() == [0, 0, 0] and r2.tolist() == [1]
    rec = np.zeros(1, dtype=oracle.RECORD_DTYPE)
    rec["level"], rec["parent_id"] = 1, 7
    ro.release(rec)
    r3, _, _, _ = ro.route(mk([7]))                # new again: the least loaded is replica 1
    assert r3.tolist() == [1]


def test_routing_keeps_aggregation_intact():
    """Sec. 4.3: groups at or below the routing level aggregate the same on
    their replica as on one aggregator."""
    for name, L in (("factcheck", 1), ("throughput", 1), ("tot", 1)):
        s = make_stream(name, small=True)
        whole = oracle.run_stream(s, drain_every=1)
        want = {}
        for d in whole:
            for r in d.records:
                if int(r["level"]) >= L:
                    want[(int(r["level"]), int(r["parent_id"]))] = (
                        int(r["n_children"]), float(r["score"]),
                        d.payload[int(r["payload_off"]):int(r["payload_off"]) + int(r["payload_len"])].tolist(),
                        d.topk[int(r["topk_off"]):int(r["topk_off"]) + int(r["topk_n"])].tolist())
        for policy in (oracle.HASH, oracle.LEAST_LOADED):
            R = 4
            ro = oracle.RouterOracle(s.depth, L, R, policy)
            aggs = [oracle.Oracle.for_stream(s) for _ in range(R)]
            got = {}
            for b in range(s.n_batches):
                _, _, _, parts = ro.route(s.batch(b))
                for r in range(R):
                    aggs[r].push_batch(parts[r])
                    d = aggs[r].drain()
                    assert d.status == 0
                    ro.release(d.records)
                    for rec in d.records:
                        if int(rec["level"]) >= L:
                            key = (int(rec["level"]), int(rec["parent_id"]))
                            assert key not in got
                            got[key] = (int(rec["n_children"]), float(rec["score"]),
                                        d.payload[int(rec["payload_off"]):int(rec["payload_off"]) +
                                                  int(rec["payload_len"])].tolist(),
                                        d.topk[int(rec["topk_off"]):int(rec["topk_off"]) + int(rec["topk_n"])].tolist())
            for a in aggs:
                a.close()
            assert got == want, (name, policy)
