"""Oracle vs hand-worked examples (tests/golden/*.json, each citing the
paper passage it is worked from)."""
import json
import os

import numpy as np
import pytest

import oracle
from declarative import same_float
from fragments import split, to_batch

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _frags(fx):
    return [(tuple(tuple(t) for t in f["tags"]), f["tokens"], f.get("score", 0.0))
            for f in fx["fragments"]]


@pytest.mark.parametrize("name", ["factool_claims.json", "factool_docs_concat_claim.json"])
def test_golden_records(name):
    fx = json.load(open(os.path.join(GOLDEN, name)))
    o = oracle.Oracle(fx["depth"], fx["payload_op"], fx["score_op"], fx["topk_k"])
    with_score = any(s != 0 for s in fx["score_op"])
    frags = _frags(fx)
    for part, exp in zip(split(frags, fx["batches"]), fx["drains"]):
        o.push_batch(to_batch(part, fx["depth"], with_score))
        d = o.drain()
        assert d.status == exp["status"]
        assert len(d.records) == len(exp["records"])
        for got, want in zip(d.records, exp["records"]):
            for k, v in want.items():
                if k == "score":
                    assert same_float(float(got[k]), v), (k, got[k], v)
                else:
                    assert int(got[k]) == v, (k, int(got[k]), v)
        assert d.payload.tolist() == exp["payload"]
        assert [(int(p["child_index"]), float(p["score"])) for p in d.topk] == \
            [tuple(x) for x in exp["topk"]]


def test_golden_errors():
    fx = json.load(open(os.path.join(GOLDEN, "errors.json")))
    for case in fx["cases"]:
        o = oracle.Oracle(fx["depth"], fx["payload_op"], fx["score_op"], fx["topk_k"])
        frags = [(tuple(tuple(t) for t in f["tags"]), f["tokens"], 0.0) for f in case["fragments"]]
        got = []
        for part in split(frags, case["batches"]):
            b = to_batch(part, fx["depth"], False)
            if case.get("bad_offsets"):
                b["off"][1], b["off"][2] = b["off"][2], b["off"][1]
            o.push_batch(b)
            got.append(o.drain().status)
        assert got == case["status"], case["name"]


def test_host_argument_checks_do_not_latch():
    o = oracle.Oracle(2, [0, 1], [0, 0], [0, 0])
    tags = np.zeros((2, 1), dtype=np.uint64)
    # depth mismatch is rejected without poisoning the handle
    assert o.push(tags, np.array([0, 0], np.uint32), np.zeros(0, np.int32), depth=3) == oracle.EINVAL
    assert o.drain().status == oracle.OK


def test_invalid_configs():
    with pytest.raises(ValueError):
        oracle.Oracle(0, [], [], [])
    with pytest.raises(ValueError):
        oracle.Oracle(9, [0] * 9, [0] * 9, [0] * 9)
    with pytest.raises(ValueError):
        oracle.Oracle(2, [1, 1], [0, 0], [0, 0])       # two CONCAT levels
    with pytest.raises(ValueError):
        oracle.Oracle(2, [0, 1], [2, 0], [0, 0])       # TOPK with k = 0
    with pytest.raises(ValueError):
        oracle.Oracle(2, [0, 1], [2, 0], [33, 0])      # TOPK with k > 32
