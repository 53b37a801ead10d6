"""Full-size parity: every workload at its full published size, through the C ABI,
with the capacities bench.py uses.

* the oracle runs on a prefix of the stream (about two million fragments) and
  those drains must match bit for bit;
* every record of the whole run is checked against properties computed from
  the stream arrays with numpy: each group emitted exactly once, records in
  strictly increasing (completion seq, deeper level first) order, completion
  seq = the largest arrival index of the group's subtree, n_children = the
  number of distinct children;
* a seeded sample of records is recomputed independently: CONCAT payload =
  the subtree's leaves in child-index path order, MAX score = largest leaf
  score (totalOrder), TOPK pairs = numpy lexsort selection over the children's
  subtree maxima.
"""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

import oracle
import paper_2403_04311_gb300 as alto
from gen import CONCAT, S_MAX, S_TOPK, make_stream

pytestmark = [pytest.mark.gpu, pytest.mark.slow]

PREFIX_FRAGMENTS = 2_000_000
SAMPLE = 128


def bench_caps(s):
    import bench
    return bench.stream_caps(s)


def total_order_keys(x):
    u = np.asarray(x, dtype=np.float32).view(np.uint32).astype(np.int64)
    return np.where(u & 0x80000000, u ^ 0xFFFFFFFF, u | 0x80000000)


def level_groups(s, l):
    """Sorted view of level l: order of leaves by parent id, run starts."""
    pid = (s.tags[l] >> np.uint64(32)).astype(np.int64)
    order = np.argsort(pid, kind="stable")
    ps = pid[order]
    starts = np.flatnonzero(np.concatenate([[True], ps[1:] != ps[:-1]]))
    return pid, order, ps, starts


def run_gpu(s, prefix_batches, drain_every):
    caps = bench_caps(s)
    agg = alto.Aggregator(s.depth, s.payload_op, s.score_op, s.topk_k, **caps)
    drains = []
    for b in range(s.n_batches):
        db = alto.to_device(s.batch(b))
        assert agg.push(db.tags, db.off, db.payload, db.score) == alto.OK
        if b < prefix_batches or (b + 1) % drain_every == 0 or b == s.n_batches - 1:
            d = agg.drain()
            assert d.status == alto.OK, (b, d.status)
            drains.append((b, d.host()))
        del db
    agg.close()
    return drains


@pytest.mark.parametrize("name", ["tiny", "factcheck", "throughput", "tokens", "adversarial", "tot"])
def test_fullsize(name):
    s = make_stream(name)
    sizes = s.batch_sizes
    prefix = max(1, int(np.searchsorted(np.cumsum(sizes), PREFIX_FRAGMENTS, side="right")))
    prefix = min(prefix, s.n_batches)
    drain_every = 1 if s.n_batches <= 64 else 64
    drains = run_gpu(s, prefix, drain_every)

    # -- oracle on the prefix, bit for bit
    o = oracle.Oracle.for_stream(s)
    for b in range(prefix):
        o.push_batch(s.batch(b))
        od = o.drain()
        gb, (rec, pay, tk) = drains[b]
        assert gb == b
        assert np.array_equal(rec.view(np.uint8), od.records.view(np.uint8)), f"{name} batch {b} records"
        assert np.array_equal(pay, od.payload), f"{name} batch {b} payload"
        assert np.array_equal(tk.view(np.uint8), od.topk.view(np.uint8)), f"{name} batch {b} top-k"
    o.close()

    # -- properties over the whole run
    recs = np.concatenate([r for _, (r, _, _) in drains])
    lv = recs["level"].astype(np.int64)
    cs = recs["completion_seq"].astype(np.int64)
    order_key = cs * 16 + (15 - lv)
    assert np.all(np.diff(order_key) > 0), "records out of (seq, deeper-first) order"
    D = s.depth
    total_groups = 0
    rng = np.random.default_rng(123)
    cids = [(s.tags[l] & np.uint64(0x7FFFFFFF)).astype(np.int64) for l in range(D)]
    score_keys = total_order_keys(s.score) if s.score is not None else None
    # index records by (level, parent id) and remember which drain holds them
    rec_drain = np.concatenate([np.full(len(r), k) for k, (_, (r, _, _)) in enumerate(drains)])
    for l in range(D):
        pid, order, ps, starts = level_groups(s, l)
        ends = np.concatenate([starts[1:], [len(ps)]])
        gids = ps[starts]
        total_groups += len(gids)
        sel = lv == l
        rl = recs[sel]
        rdr = rec_drain[sel]
        assert len(rl) == len(gids), f"{name} level {l}: {len(rl)} records for {len(gids)} groups"
        rp = rl["parent_id"].astype(np.int64)
        ri = np.argsort(rp)
        assert np.array_equal(rp[ri], gids), f"{name} level {l}: groups emitted once each"
        # completion seq and child count per group
        max_seq = np.maximum.reduceat(order, starts)
        assert np.array_equal(rl["completion_seq"][ri].astype(np.int64), max_seq)
        key = np.sort(ps * (1 << 31) + cids[l][order])  # groups stay in parent order
        distinct = np.concatenate([[True], key[1:] != key[:-1]])
        nch = np.add.reduceat(distinct.astype(np.int64), starts)
        assert np.array_equal(rl["n_children"][ri].astype(np.int64), nch)
        # sampled recomputation
        pick = rng.choice(len(gids), size=min(SAMPLE, len(gids)), replace=False)
        for g in pick:
            r = rl[ri[g]]
            dk = rdr[ri[g]]
            leaves = order[starts[g]:ends[g]]
            if s.payload_op[l] == CONCAT:
                path = tuple(cids[q][leaves] for q in reversed(range(l, D)))
                lo = leaves[np.lexsort(path)]
                want = np.concatenate([s.payload[s.off[i]:s.off[i + 1]] for i in lo])
                _, (_, pay, _) = drains[dk]
                got = pay[int(r["payload_off"]):int(r["payload_off"]) + int(r["payload_len"])]
                assert np.array_equal(got, want), f"{name} level {l} group {gids[g]} payload"
            if s.score_op[l] in (S_MAX, S_TOPK):
                best = s.score[leaves][np.argmax(score_keys[leaves])]
                assert np.float32(r["score"]).view(np.uint32) == np.float32(best).view(np.uint32)
            if s.score_op[l] == S_TOPK:
                child = cids[l][leaves]
                uc, inv = np.unique(child, return_inverse=True)
                cmax = np.full(len(uc), -1, dtype=np.int64)
                np.maximum.at(cmax, inv, score_keys[leaves])
                k = int(s.topk_k[l])
                sel_c = np.lexsort((uc, -cmax))[:k]
                _, (_, _, tk) = drains[dk]
                got = tk[int(r["topk_off"]):int(r["topk_off"]) + int(r["topk_n"])]
                assert got["child_index"].astype(np.int64).tolist() == uc[sel_c].tolist()
    assert total_groups == len(recs)
