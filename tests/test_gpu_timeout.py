"""A device wait that runs out: ETIMEOUT, latched, and a usable context after.

Every look-back wait on the device is capped at spin_limit polls; a wait that
reaches the cap records ALTO_ETIMEOUT, sets the batch's abort flag (every
later kernel of the batch returns at once) and the push's work ends.  No
input makes a wait run out by itself, so the test uses ALTO_FLAG_TEST_STALL:
each wait then polls a predecessor's descriptor that nothing publishes.  The
batches are built so that the first scan (or sort) with a wait has more than
one tile.  Checked: the drain returns ETIMEOUT within seconds, later pushes
and drains return it too, destroy succeeds, and a fresh handle on the same
device then aggregates a stream bit for bit like the oracle."""
import time

import numpy as np
import pytest

torch = pytest.importorskip("torch")

import paper_2403_04311_gb300 as alto
from fragments import to_batch
from gen import make_stream
from gpu_harness import assert_same, run_both_stream

pytestmark = pytest.mark.gpu


def _one_group(n, scored):
    """Depth 1: one group with children 0..n-1 in one batch (reversed order),
    one token each; it completes, so its n dense child slots are scanned."""
    frags = [(((7, c, c == n - 1),), [c % 50257], float(c % 13) - 6.0) for c in reversed(range(n))]
    return to_batch(frags, 1, scored)


@pytest.mark.parametrize("form", ["dense_scan", "radix_sort"])
def test_stalled_wait_reports_etimeout_and_the_context_stays_usable(form):
    n = 10_000  # three 4,096-element scan tiles, three 4,096-key sort tiles
    if form == "dense_scan":
        # sort-free leaf level: the dense child-slot scan is the first multi-tile scan
        ops = dict(depth=1, payload_op=[1], score_op=[0], topk_k=[0])
        bt = _one_group(n, False)
    else:
        # top-k at the leaf parent: the leaf level is sorted by table slot
        ops = dict(depth=1, payload_op=[1], score_op=[2], topk_k=[4])
        bt = _one_group(n, True)
    caps = dict(max_batch_fragments=n, max_batch_payload=n, max_open_groups=1024, arena_elems=1 << 16,
                out_records=1024, out_payload_elems=2 * n, out_topk=1024, max_emit_children=2 * n,
                spin_limit=256, test_stall=True)
    agg = alto.Aggregator(ops["depth"], ops["payload_op"], ops["score_op"], ops["topk_k"], **caps)
    try:
        db = alto.to_device(bt)
        t0 = time.perf_counter()
        assert agg.push(db.tags, db.off, db.payload, db.score) == alto.OK  # enqueue only
        d = agg.drain()
        elapsed = time.perf_counter() - t0
        assert d.status == alto.ETIMEOUT
        assert elapsed < 10.0, elapsed
        # latched: later pushes and drains report it, nothing runs
        assert agg.push(db.tags, db.off, db.payload, db.score) == alto.ETIMEOUT
        assert agg.drain().status == alto.ETIMEOUT
    finally:
        agg.close()  # destroy succeeds on a poisoned handle
    torch.cuda.synchronize()
    # the context is still usable: a fresh handle matches the oracle
    s = make_stream("factcheck", small=True)
    o, g = run_both_stream(s)
    assert_same(o, g, "after a timed-out handle")


def test_stall_flag_changes_nothing_without_a_wait():
    """A batch whose scans and sorts all fit one tile never waits, so the
    hook leaves it alone: same records as without the flag."""
    bt = _one_group(3000, False)
    caps = dict(max_batch_fragments=3000, max_batch_payload=3000, max_open_groups=1024,
                arena_elems=1 << 16, out_records=1024, out_payload_elems=6000, out_topk=1024,
                max_emit_children=4000, spin_limit=256)
    out = []
    for stall in (False, True):
        agg = alto.Aggregator(1, [1], [0], [0], test_stall=stall, **caps)
        db = alto.to_device(bt)
        assert agg.push(db.tags, db.off, db.payload, db.score) == alto.OK
        d = agg.drain()
        assert d.status == alto.OK
        out.append(d.host())
        agg.close()
    for a, b in zip(out[0], out[1]):
        assert np.array_equal(np.asarray(a).view(np.uint8), np.asarray(b).view(np.uint8))
