"""The split placement on the GPU, bit for bit against the oracle through the
C ABI.

With CONCAT at the leaf parent and the sort-free leaf level, a push forks
after the leaf finalize into three streams:
- the completing leaf parents' payload path (their ranks among themselves,
  offsets, dense placement, length scan, gather) on a second stream;
- the open groups' arena copies on a third;
- the upper levels, the record scans, the records and the sweep on the
  push's stream.
Replayed push graphs hold the same work as parallel branches.  Only leaf
parents carry payload, and their emission order among themselves is their
completion order (Sec. 3.2, Sec. 4.2), so the payload offsets need nothing
from the levels above.

The cases:
- streams cut so that one handle replays graphs for some pushes and launches
  others kernel by kernel;
- each output capacity overflowing in exactly one batch of a stream drained
  after every batch.  That batch reports ENOSPC, every earlier drain matches
  the oracle, and the error stays latched;
- the golden error cases with every kernel launched by itself.
"""
import dataclasses
import json
import os

import numpy as np
import pytest

torch = pytest.importorskip("torch")

import paper_2403_04311_gb300 as alto
from fragments import split, to_batch
from gen import make_stream
from gpu_harness import assert_same, run_gpu_batches, run_oracle_batches, small_caps, stream_caps

pytestmark = pytest.mark.gpu

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _recut(s, sizes):
    assert sum(sizes) == s.n
    return dataclasses.replace(s, batch_sizes=np.asarray(sizes, dtype=np.int64))


def _run(s, caps, direct=False):
    batches = [s.batch(b) for b in range(s.n_batches)]
    caps = dict(caps, direct_launch=direct)
    _, g = run_gpu_batches(s.depth, s.payload_op, s.score_op, s.topk_k, batches, caps)
    o = run_oracle_batches(s.depth, s.payload_op, s.score_op, s.topk_k, batches)
    return o, g


# pushes above 128K fragments launch kernel by kernel, the others replay a
# graph of their size class: both kinds on one handle, in either order
@pytest.mark.parametrize("name,sizes", [
    ("factcheck", [20_000, 140_000, 3_000, 150_000, 40_955]),
    ("factcheck", [150_000, 1, 129_000, 74_954]),
    ("throughput", [130_000, 5_000, 65_000]),
])
def test_graph_and_direct_pushes_on_one_handle(name, sizes):
    s = _recut(make_stream(name, small=(name == "throughput")), sizes)
    o, g = _run(s, stream_caps(s))
    assert all(d.status == alto.OK for d in o)
    assert_same(o, g, f"{name} {sizes}")


def _per_batch(o, s):
    """Per drained batch: records, payload elements, dense slots (children of
    the completing leaf parents) and top-k pairs."""
    M = s.depth - 1
    out = []
    for d in o:
        r = d.records
        out.append({
            "out_records": len(r),
            "out_payload_elems": len(d.payload),
            "max_emit_children": int(r["n_children"][r["level"] == M].astype(np.int64).sum()),
            "out_topk": int(r["topk_n"].astype(np.int64).sum()),
        })
    return out


@pytest.mark.parametrize("direct", [False, True])
@pytest.mark.parametrize("cap", ["out_records", "out_payload_elems", "max_emit_children", "out_topk"])
def test_each_capacity_overflows_in_one_batch(cap, direct):
    s = make_stream("factcheck", small=True)   # TOPK above, CONCAT at the leaf parent
    batches = [s.batch(b) for b in range(s.n_batches)]
    o = run_oracle_batches(s.depth, s.payload_op, s.score_op, s.topk_k, batches)
    assert all(d.status == alto.OK for d in o)
    use = [u[cap] for u in _per_batch(o, s)]
    limit = max(max(use) - 1, 1)
    assert max(use) > limit, f"{cap}: no batch needs more than one ({use})"
    first = next(b for b, u in enumerate(use) if u > limit)
    caps = dict(stream_caps(s), direct_launch=direct)
    caps[cap] = limit
    _, g = run_gpu_batches(s.depth, s.payload_op, s.score_op, s.topk_k, batches, caps)
    assert_same(o[:first], g[:first], f"{cap} before batch {first}")
    assert [x[0] for x in g[first:]] == [alto.ENOSPC] * (len(g) - first), f"{cap}: {[x[0] for x in g]}"


def test_golden_errors_kernel_by_kernel():
    """The hand-written error cases with every kernel launched by itself: the
    placement's streams stand down on errors raised before they fork, and the
    reported class is the same as with graph replay."""
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
        caps = dict(small_caps(8, 16, fx["depth"]), direct_launch=True)
        _, g = run_gpu_batches(fx["depth"], fx["payload_op"], fx["score_op"], fx["topk_k"], batches, caps)
        assert [d[0] for d in g] == case["status"], case["name"]
