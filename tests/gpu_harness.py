"""Run streams through the CUDA library and the oracle, and compare drains
bit for bit (test infrastructure)."""
from __future__ import annotations

import numpy as np

import oracle
import paper_2403_04311_gb300 as alto


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
