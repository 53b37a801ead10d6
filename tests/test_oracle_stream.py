"""Streaming release in the oracle, against facts it does not compute itself.

Sec. 3.2: the outputs of a pmap are put back in their original order and
passed on as a stream.  With streaming release, an open CONCAT group emits,
after each batch, the children 0..r-1 that are complete and not yet released
as a partial record; its final record carries the rest.

* a hand-worked stream of one group (partial, nothing, final);
* conservation: per CONCAT group, the payloads of its partial records and of
  its final record, in record order, are the payload the group's one record
  has without streaming release; the final record keeps every other field;
* records at the other levels are those of the run without streaming;
* partial records: n_children rises strictly, stays below the final count,
  carries no score or top-k, and the seq is the latest arrival among the
  released leaves (checked from the tags, for the leaf-parent CONCAT level);
* every drain is in strictly increasing (seq, deeper level first) order;
* the same at a CONCAT level above the leaf parent.
(The brute-force test checks every field against the non-incremental
definition on small trees.)
"""
import dataclasses

import numpy as np
import pytest

import oracle
from fragments import pack
from gen import make_stream


def _batch(frags, depth):
    n = len(frags)
    tags = np.zeros((depth, n), np.uint64)
    off = np.zeros(n + 1, np.uint32)
    toks = []
    for i, (t, tok) in enumerate(frags):
        for l in range(depth):
            tags[l, i] = pack(*t[l])
        off[i + 1] = off[i] + len(tok)
        toks.extend(tok)
    return dict(n=n, tags=tags, off=off, payload=np.asarray(toks, np.int32), score=None)


def test_hand_worked_stream():
    # one query (level 0, id 1) with one stream (level 1, id 9) of 4 pieces
    def f(c, last=False):
        return (((1, 0, True), (9, c, last)), [10 * c, 10 * c + 1])
    o = oracle.Oracle(2, [0, 1], [0, 0], [0, 0], stream_release=True)
    o.push_batch(_batch([f(1), f(0)], 2))          # seq 0, 1: children 0, 1 in order
    d = o.drain()
    assert d.status == 0 and len(d.records) == 1
    r = d.records[0]
    assert (int(r["level"]), int(r["parent_id"]), int(r["n_children"]), int(r["completion_seq"]),
            int(r["ops"])) == (1, 9, 2, 1, 0x81)
    assert d.payload.tolist() == [0, 1, 10, 11]
    o.push_batch(_batch([f(3, True)], 2))          # seq 2: child 2 still missing
    d = o.drain()
    assert d.status == 0 and len(d.records) == 0
    o.push_batch(_batch([f(2)], 2))                # seq 3: the group and the query complete
    d = o.drain()
    assert d.status == 0
    got = [(int(r["level"]), int(r["parent_id"]), int(r["n_children"]), int(r["completion_seq"]), int(r["ops"]))
           for r in d.records]
    assert got == [(1, 9, 4, 3, 0x01), (0, 1, 1, 3, 0x00)]
    assert d.payload.tolist() == [20, 21, 30, 31]
    o.close()


def _records(drains):
    """Per drain: list of (record fields, payload, topk)."""
    out = []
    for d in drains:
        assert d.status == 0
        rows = []
        for r in d.records:
            pay = d.payload[int(r["payload_off"]):int(r["payload_off"]) + int(r["payload_len"])].tolist()
            tk = d.topk[int(r["topk_off"]):int(r["topk_off"]) + int(r["topk_n"])].tolist()
            rows.append((r, pay, tk))
        out.append(rows)
    return out


def _key(r):
    return (int(r["completion_seq"]), int(r["level"]), int(r["parent_id"]), int(r["n_children"]),
            int(r["ops"]), np.float32(r["score"]).view(np.uint32).item())


def _check_stream(s):
    M = list(s.payload_op).index(1)
    plain = _records(oracle.run_stream(s, drain_every=1))
    strm = _records(oracle.run_stream(s, drain_every=1, stream_release=True))
    assert len(plain) == len(strm)
    whole = {}
    for rows in plain:
        for r, pay, tk in rows:
            if int(r["level"]) == M:
                whole[int(r["parent_id"])] = (r, pay, tk)
    got_pay, last_n, n_partial = {}, {}, 0
    for b, (prow, srow) in enumerate(zip(plain, strm)):
        # the other levels are untouched
        other_p = [(_key(r), pay, tk) for r, pay, tk in prow if int(r["level"]) != M]
        other_s = [(_key(r), pay, tk) for r, pay, tk in srow if int(r["level"]) != M]
        assert other_p == other_s, b
        keys = [(int(r["completion_seq"]), -int(r["level"])) for r, _, _ in srow]
        assert all(a < c for a, c in zip(keys, keys[1:])), b
        for r, pay, tk in srow:
            if int(r["level"]) != M:
                continue
            p = int(r["parent_id"])
            got_pay.setdefault(p, []).extend(pay)
            if int(r["ops"]) & 0x80:
                n_partial += 1
                assert int(r["ops"]) == 0x81 and float(r["score"]) == 0.0 and tk == []
                assert int(r["n_children"]) > last_n.get(p, 0)
                last_n[p] = int(r["n_children"])
            else:
                w, _wpay, wtk = whole[p]
                assert _key(r) == _key(w) and tk == wtk
                assert int(r["n_children"]) > last_n.get(p, -1)
                last_n[p] = None
    assert set(whole) <= set(got_pay)
    for p, (_w, wpay, _) in whole.items():
        assert got_pay[p] == wpay, p
    return n_partial


def _partial_seq_from_tags(s):
    """Leaf-parent CONCAT level: a partial record's seq is the latest arrival
    index among the leaves it releases (recomputed from the tags)."""
    D = s.depth
    leaf_pid = (s.tags[D - 1] >> np.uint64(32)).astype(np.int64)
    leaf_c = (s.tags[D - 1] & np.uint64(0x7FFFFFFF)).astype(np.int64)
    arrival = {(int(p), int(c)): i for i, (p, c) in enumerate(zip(leaf_pid, leaf_c))}
    strm = oracle.run_stream(s, drain_every=1, stream_release=True)
    rel = {}
    checked = 0
    for d in strm:
        for r in d.records:
            if int(r["level"]) != D - 1 or not (int(r["ops"]) & 0x80):
                continue
            p, n = int(r["parent_id"]), int(r["n_children"])
            r0 = rel.get(p, 0)
            assert int(r["completion_seq"]) == max(arrival[(p, c)] for c in range(r0, n))
            rel[p] = n
            checked += 1
    return checked


@pytest.mark.parametrize("name", ["tiny", "factcheck", "throughput", "tokens", "tot", "adversarial"])
def test_stream_release_invariants(name):
    s = make_stream(name, small=True)
    n_partial = _check_stream(s)
    assert n_partial > 0 or s.n_batches == 1
    if list(s.payload_op).index(1) == s.depth - 1:
        assert _partial_seq_from_tags(s) == n_partial


@pytest.mark.parametrize("name,m", [("factcheck", 1), ("factcheck", 2), ("tot", 1), ("throughput", 0)])
def test_stream_release_upper_concat(name, m):
    s = make_stream(name, small=True)
    po = [0] * s.depth
    po[m] = 1
    s = dataclasses.replace(s, payload_op=tuple(po))
    _check_stream(s)


def test_stream_release_needs_concat():
    with pytest.raises(ValueError):
        oracle.Oracle(2, [0, 0], [0, 0], [0, 0], stream_release=True)
