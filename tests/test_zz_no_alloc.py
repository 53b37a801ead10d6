"""The allocation-free one-shot entry point against the oracle and the regular path.

alto_agg_oneshot_noalloc exists for callers that may not allocate device
memory (a framework that already reserved the device's free memory for its
own pool, a real-time path that cannot take cudaMalloc's synchronisation, a
plug-in loaded without an allocator).  It works out of a static device array
and writes into buffers the caller owns.  Each batch goes through it twice in
a row, and must give exactly the records, payload and top-k pairs of the
oracle and of create + push_batch + drain on a fresh handle (exact equality:
the results are integers and copied floats).  The batches follow one another
with different depths, CONCAT levels and k, so that each call finds the
static array laid out differently by the call before; one of them carries
token ids 1..64, values the arrays read by epoch stamp could mistake for a
stamp if a call did not clear them.  This file is collected last on purpose."""
import dataclasses

import numpy as np
import pytest

torch = pytest.importorskip("torch")

import oracle
import paper_2403_04311_gb300 as alto
from gen import make_stream
from gen.streams import make_factcheck

pytestmark = pytest.mark.gpu


def _regular(s, bt, caps):
    agg = alto.Aggregator(s.depth, s.payload_op, s.score_op, s.topk_k, **caps)
    db = alto.to_device(bt)
    assert agg.push(db.tags, db.off, db.payload, db.score) == alto.OK
    d = agg.drain()
    assert d.status == alto.OK
    rec, pay, tk = d.host()
    agg.close()
    return rec, pay, tk


def _oneshot(s, bt, cap_rec=8192, cap_pay=1 << 18, cap_topk=8192):
    cfg = alto.make_config(s.depth, s.payload_op, s.score_op, s.topk_k,
                           max_batch_fragments=0, max_batch_payload=0)
    db = alto.to_device(bt)
    b = alto.alto_batch()
    b.n = bt["n"]
    b.depth = s.depth
    b.tags = db.tags.data_ptr()
    b.payload_off = db.off.data_ptr()
    b.n_payload = int(db.payload.numel())
    b.payload = db.payload.data_ptr()
    b.score = db.score.data_ptr() if db.score is not None else None
    # output buffers belong to the caller (the test); the entry point allocates nothing
    rec = torch.zeros(cap_rec * 48, dtype=torch.uint8, device="cuda")
    pay = torch.zeros(cap_pay, dtype=torch.int32, device="cuda")
    tk = torch.zeros(cap_topk * 8, dtype=torch.uint8, device="cuda")
    counts = torch.zeros(4, dtype=torch.int64, device="cuda")
    stream = torch.cuda.current_stream().cuda_stream
    st = alto.alto_agg_oneshot_noalloc(cfg, b, rec.data_ptr(), cap_rec, pay.data_ptr(), cap_pay,
                                       tk.data_ptr(), cap_topk, counts.data_ptr(), stream)
    assert st == alto.OK
    torch.cuda.synchronize()
    c = counts.cpu().numpy()
    assert c[0] == alto.OK, c
    nr, npay, ntk = int(c[1]), int(c[2]), int(c[3])
    return (rec[:nr * 48].cpu().numpy().view(alto.RECORD_DTYPE), pay[:npay].cpu().numpy(),
            tk[:ntk * 8].cpu().numpy().view(alto.PAIR_DTYPE))


def _oracle(s, bt):
    o = oracle.Oracle.for_stream(s)
    assert o.push_batch(bt) == oracle.OK
    d = o.drain()
    o.close()
    assert d.status == oracle.OK
    return d.records, d.payload, d.topk


def _cases():
    tiny = make_stream("tiny64")
    # token ids 1..64: small integers like the epochs the static array's
    # stamped slots are compared with
    tiny_small = dict(tiny.batch(0))
    tiny_small["payload"] = (tiny_small["payload"] % 64 + 1).astype(np.int32)
    # depth 4 with top-k and max levels, whole stream in one batch
    fact = make_factcheck(n_responses=8, batch=4096)
    assert fact.n_batches == 1
    # the same batch with the concatenation two levels above the fragments
    fact_up = dataclasses.replace(fact, payload_op=(0, 1, 0, 0))
    a, b, c = (tiny, tiny_small), (fact, fact.batch(0)), (fact_up, fact_up.batch(0))
    # every layout after another one, and each again after a change
    return [a, b, c, a, c, b, a]


def _same(got, want):
    assert np.array_equal(got[0].view(np.uint8), want[0].view(np.uint8))
    assert np.array_equal(got[1], want[1])
    assert np.array_equal(got[2].view(np.uint8), want[2].view(np.uint8))


def test_oneshot_noalloc_matches_oracle_and_regular_path_twice_in_a_row():
    for s, bt in _cases():
        assert bt["n"] <= 4096 and bt["n"] * s.depth <= 16384
        caps = dict(max_batch_fragments=bt["n"], max_batch_payload=int(bt["payload"].size),
                    max_open_groups=1 << 15, arena_elems=1 << 22, out_records=1 << 15,
                    out_payload_elems=1 << 18, out_topk=1 << 15, max_emit_children=1 << 14)
        want = _oracle(s, bt)
        assert len(want[0]) > 0
        _same(_regular(s, bt, caps), want)
        first = _oneshot(s, bt)
        second = _oneshot(s, bt)
        _same(first, want)
        _same(second, want)


def test_oneshot_noalloc_rejects_oversize_batches():
    s = make_stream("tiny")   # one batch of 4,096 fragments at depth 2: fits
    bt = s.batch(0)
    big = make_stream("factcheck", small=True)
    cfg = alto.make_config(big.depth, big.payload_op, big.score_op, big.topk_k,
                           max_batch_fragments=0, max_batch_payload=0)
    b = alto.alto_batch()
    b.n = 5000            # above the 4,096-fragment limit
    b.depth = big.depth
    b.n_payload = 0
    counts = torch.zeros(4, dtype=torch.int64, device="cuda")
    st = alto.alto_agg_oneshot_noalloc(cfg, b, 0, 0, 0, 0, 0, 0, counts.data_ptr(), 0)
    assert st == alto.ENOSPC
    got = _oneshot(s, bt)
    assert len(got[0]) > 0
