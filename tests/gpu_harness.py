"""Run streams through the CUDA library and the oracle, and compare drains
bit for bit (test infrastructure)."""
from __future__ import annotations

import numpy as np

import oracle
import paper_2403_04311_gb300 as alto


def small_caps(n, payload, depth, k=8):
    """Capacities for hand-built streams of a few thousand fragments."""
    return dict(max_batch_fragments=max(n, 1), max_batch_payload=max(payload, 1),
                max_open_groups=4096, arena_elems=1 << 16, out_records=4096,
                out_payload_elems=1 << 14, out_topk=4096, max_emit_children=4096)


def stream_caps(s, arena_factor=4, stream_release=False):
    """Capacities that hold a whole generated stream (with streaming release,
    every fragment may also bring one partial record)."""
    D, n = s.depth, s.n
    groups = sum(len(np.unique(s.tags[l] >> np.uint64(32))) for l in range(D))
    st = s.batch_starts()
    pay_per_batch = [int(s.off[st[b + 1]] - s.off[st[b]]) for b in range(s.n_batches)]
    kmax = max(list(s.topk_k) + [1])
    return dict(
        max_batch_fragments=int(max(s.batch_sizes)),
        max_batch_payload=max(1, max(pay_per_batch)),
        max_open_groups=min(groups + 1024, 1 << 25),
        arena_elems=min(arena_factor * (int(s.payload.size) + 2 * n) + 64 * groups + (1 << 16),
                        (1 << 32) - 1),
        out_records=groups + 16 + (n if stream_release else 0),
        out_payload_elems=int(s.payload.size) + 16,
        out_topk=groups * kmax + 16,
        max_emit_children=n + 16,
    )


def gpu_drain_host(d):
    if d.status != alto.OK:
        return d.status, None, None, None
    rec, pay, tk = d.host()
    return d.status, rec, pay, tk


def run_gpu_batches(depth, payload_op, score_op, topk_k, batches, caps, drain_after=None):
    """batches: list of batch dicts (host).  Returns (push statuses, drains)."""
    agg = alto.Aggregator(depth, payload_op, score_op, topk_k, **caps)
    drains, pushes = [], []
    try:
        for b, bt in enumerate(batches):
            db = alto.to_device(bt)
            pushes.append(agg.push(db.tags, db.off, db.payload, db.score))
            if drain_after is None or drain_after[b] or b == len(batches) - 1:
                drains.append(gpu_drain_host(agg.drain()))
    finally:
        agg.close()
    return pushes, drains


def run_oracle_batches(depth, payload_op, score_op, topk_k, batches, drain_after=None, stream_release=False):
    o = oracle.Oracle(depth, payload_op, score_op, topk_k, stream_release=stream_release)
    out = []
    for b, bt in enumerate(batches):
        o.push_batch(bt)
        if drain_after is None or drain_after[b] or b == len(batches) - 1:
            out.append(o.drain())
    o.close()
    return out


def assert_same(oracle_drains, gpu_drains, ctx=""):
    assert len(oracle_drains) == len(gpu_drains), ctx
    for k, (od, (st, rec, pay, tk)) in enumerate(zip(oracle_drains, gpu_drains)):
        assert st == od.status, f"{ctx} drain {k}: gpu status {st} oracle {od.status}"
        if st != alto.OK:
            continue
        assert len(rec) == len(od.records), f"{ctx} drain {k}: {len(rec)} vs {len(od.records)} records"
        if not np.array_equal(rec.view(np.uint8), od.records.view(np.uint8)):
            bad = np.flatnonzero((rec.view(np.uint8).reshape(-1, 48) !=
                                  od.records.view(np.uint8).reshape(-1, 48)).any(1))
            i = int(bad[0])
            raise AssertionError(f"{ctx} drain {k}: record {i} differs: gpu {rec[i]} oracle {od.records[i]}")
        assert np.array_equal(pay, od.payload), f"{ctx} drain {k}: payload differs"
        assert np.array_equal(tk.view(np.uint8), od.topk.view(np.uint8)), f"{ctx} drain {k}: top-k differs"


def run_both_stream(s, drain_every=1, caps=None, stream_release=False):
    batches = [s.batch(b) for b in range(s.n_batches)]
    da = [((b + 1) % drain_every == 0) for b in range(s.n_batches)]
    caps = dict(caps or stream_caps(s, stream_release=stream_release))
    if stream_release:
        caps["stream_release"] = True
    _, g = run_gpu_batches(s.depth, s.payload_op, s.score_op, s.topk_k, batches, caps, da)
    o = run_oracle_batches(s.depth, s.payload_op, s.score_op, s.topk_k, batches, da, stream_release)
    return o, g


def route_release_and_aggregate(s, L=1, R=4, max_flows=0):
    """Route stream s at level L into R GPU aggregators, release completed
    flows from the aggregators' device records, and check it against the
    oracle router and one oracle aggregator over the whole stream: replicas
    match batch by batch, and every group at level >= L gets the record the
    whole stream gives it (Sec. 4.3)."""
    bsz = int(max(s.batch_sizes))
    pay = int(max(s.off[b1] - s.off[b0] for b0, b1 in zip(s.batch_starts()[:-1], s.batch_starts()[1:])))
    rt = alto.Router(s.depth, L, R, alto.ROUTE_LEAST_LOADED, max_batch_fragments=bsz, max_batch_payload=pay,
                     max_flows=max_flows, with_score=s.score is not None)
    ro = oracle.RouterOracle(s.depth, L, R, oracle.LEAST_LOADED)
    caps = stream_caps(s)
    aggs = [alto.Aggregator(s.depth, s.payload_op, s.score_op, s.topk_k, **caps) for _ in range(R)]
    whole = oracle.run_stream(s, drain_every=1)
    want = {}
    for d in whole:
        for r in d.records:
            if int(r["level"]) >= L:
                want[(int(r["level"]), int(r["parent_id"]))] = (
                    int(r["n_children"]), d.payload[int(r["payload_off"]):int(r["payload_off"]) + int(r["payload_len"])].tolist())
    got = {}
    for b in range(s.n_batches):
        bt = s.batch(b)
        db = alto.to_device(bt)
        assert rt.route(db.tags, db.off, db.payload, db.score) == alto.OK
        st, fo, po = rt.counts()
        assert st == alto.OK
        replica, _, _, _ = ro.route(bt)
        rep_d, _, parts = rt.outputs(fo, po)
        assert np.array_equal(rep_d.cpu().numpy(), replica)
        for r in range(R):
            t, o, p, sc = parts[r]
            if t.shape[1]:
                assert aggs[r].push(t.contiguous(), o, p, sc) == alto.OK
            d = aggs[r].drain()
            assert d.status == alto.OK
            rec, payl, _ = d.host()
            if len(rec):
                assert rt.release(d.records.data_ptr(), len(rec)) == alto.OK
            ro.release(rec)
            for x in rec:
                if int(x["level"]) >= L:
                    got[(int(x["level"]), int(x["parent_id"]))] = (
                        int(x["n_children"]), payl[int(x["payload_off"]):int(x["payload_off"]) + int(x["payload_len"])].tolist())
    for a in aggs:
        a.close()
    rt.close()
    assert got == want


def route_stream_vs_oracle(s, level, R, policy, batches=None, max_flows=0):
    """Route the batches of stream s and compare, batch by batch, each
    fragment's replica, the stable partition, the replica offsets and every
    replica's sub-batch with the routing oracle's."""
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
