"""Oracle vs the non-incremental declarative evaluation, by enumeration.

Small trees (depth 1-3, fanout 1-3 per level, at most 7 leaves): every
arrival order and every batch cut for trees of up to 4 leaves, a seeded
sample of both for larger ones; every choice of the CONCAT level; MAX and
TOPK (k = 1, 2) with tied scores and signed zeros.  Then the same with one
defect injected (duplicate, moved last flag, changed parent tag or child
index), where only the status has to agree."""
import itertools
import random

import pytest

import oracle
from declarative import evaluate, same_float
from fragments import split, to_batch, tree_fragments

SCORES = [-1.0, -0.0, 0.0, 0.5, 0.5, 2.0, -3.5]


def shapes(depth, max_leaves=7):
    if depth == 1:
        return [k for k in (1, 2, 3)]
    out = []
    sub = shapes(depth - 1, max_leaves)
    for k in (1, 2, 3):
        for combo in itertools.product(sub, repeat=k):
            if count_leaves(list(combo)) <= max_leaves:
                out.append(list(combo))
    return out


def count_leaves(s):
    return s if isinstance(s, int) else sum(count_leaves(x) for x in s)


def ops_variants(depth, rng):
    """(payload_op, score_op, topk_k) choices: each CONCAT level (or none)
    with a random score-op assignment."""
    out = []
    for m in list(range(depth)) + [None]:
        po = [1 if l == m else 0 for l in range(depth)]
        so = [rng.choice([0, 1, 2]) for _ in range(depth)]
        kk = [rng.choice([1, 2]) if s == 2 else 0 for s in so]
        out.append((po, so, kk))
    return out


def cuts(n):
    for mask in range(1 << (n - 1)):
        sizes, cur = [], 1
        for i in range(n - 1):
            if mask >> i & 1:
                sizes.append(cur)
                cur = 1
            else:
                cur += 1
        sizes.append(cur)
        yield sizes


def run_oracle(depth, po, so, kk, frags, sizes, corrupt=None, stream_release=False):
    o = oracle.Oracle(depth, po, so, kk, stream_release=stream_release)
    with_score = any(s != 0 for s in so)
    res = []
    for b, part in enumerate(split(frags, sizes)):
        bt = to_batch(part, depth, with_score)
        if corrupt is not None and corrupt == b:
            bt["off"][-1] = bt["off"][-1] + 1  # beyond the payload slice
        o.push_batch(bt)
        res.append(o.drain())
    o.close()
    return res


def compare(depth, po, so, kk, frags, sizes, status_only=False, stream_release=False):
    want = evaluate(depth, po, so, kk, frags, sizes, stream_release=stream_release)
    got = run_oracle(depth, po, so, kk, frags, sizes, stream_release=stream_release)
    for b, ((st, recs, pay, topk), d) in enumerate(zip(want, got)):
        assert d.status == st, (b, d.status, st, frags, sizes)
        if status_only or st != 0:
            continue
        assert len(d.records) == len(recs), (b, frags, sizes)
        for r, w in zip(d.records, recs):
            for k, v in w.items():
                if k == "score":
                    assert same_float(float(r[k]), v), (k, r[k], v)
                else:
                    assert int(r[k]) == v, (k, int(r[k]), v, frags, sizes)
        assert d.payload.tolist() == pay
        assert len(d.topk) == len(topk)
        for p, (c, s) in zip(d.topk, topk):
            assert int(p["child_index"]) == c and same_float(float(p["score"]), s)


def _cases(depth, exhaustive_upto=4, samples=12, seed=0):
    rng = random.Random(seed + depth)
    for shape in shapes(depth):
        frags = tree_fragments(shape, score_fn=lambda k: SCORES[k % len(SCORES)])
        n = len(frags)
        for po, so, kk in ops_variants(depth, rng):
            if n <= exhaustive_upto:
                orders = list(itertools.permutations(range(n)))
                combos = [(p, c) for p in orders for c in cuts(n)]
                if len(combos) > 200:
                    combos = rng.sample(combos, 200)
            else:
                combos = []
                for _ in range(samples):
                    p = list(range(n))
                    rng.shuffle(p)
                    c = rng.choice(list(cuts(n)))
                    combos.append((p, c))
            for p, c in combos:
                yield [frags[i] for i in p], c, po, so, kk


@pytest.mark.parametrize("depth", [1, 2, 3])
def test_bruteforce_valid(depth):
    count = 0
    for frags, sizes, po, so, kk in _cases(depth):
        compare(depth, po, so, kk, frags, sizes)
        count += 1
    assert count > 50


@pytest.mark.parametrize("depth", [1, 2, 3])
def test_bruteforce_stream_release(depth):
    """Streaming release at every CONCAT level: partial records per batch
    against the prefix of complete children recomputed from scratch."""
    count = partial = 0
    for frags, sizes, po, so, kk in _cases(depth, samples=8, seed=31):
        if 1 not in po:
            continue
        compare(depth, po, so, kk, frags, sizes, stream_release=True)
        want = evaluate(depth, po, so, kk, frags, sizes, stream_release=True)
        partial += sum(1 for _st, recs, _p, _t in want for r in recs if r["ops"] & 0x80)
        count += 1
    assert count > 20 and partial > 10


def test_bruteforce_forest():
    """Two independent sources interleaved, at depths 2 and 3."""
    rng = random.Random(7)
    pairs = [([2, 1], [1]), ([[1], [2]], [[2, 1]]), ([3], [2, 2])]
    for shape_a, shape_b in pairs:
        da = depth_of(shape_a)
        assert da == depth_of(shape_b)
        fa = tree_fragments(shape_a, id_base=100, score_fn=lambda k: SCORES[k % 7])
        fb = tree_fragments(shape_b, id_base=500, score_fn=lambda k: SCORES[(k + 3) % 7])
        frags = fa + fb
        for _ in range(60):
            p = list(range(len(frags)))
            rng.shuffle(p)
            c = rng.choice(list(cuts(len(frags))))
            for po, so, kk in ops_variants(da, rng):
                compare(da, po, so, kk, [frags[i] for i in p], c)


def depth_of(s):
    return 1 if isinstance(s, int) else 1 + depth_of(s[0])


def mutate(frags, rng):
    frags = list(frags)
    kind = rng.randrange(5)
    i = rng.randrange(len(frags))
    tags, tok, sc = frags[i]
    tags = list(tags)
    l = rng.randrange(len(tags))
    p, c, f = tags[l]
    if kind == 0:                       # duplicate a fragment later on
        j = rng.randrange(i, len(frags) + 1)
        frags.insert(j, frags[i])
        return frags
    if kind == 1:
        tags[l] = (p, c, not f)         # move / add / drop a last flag
    elif kind == 2:
        tags[l] = (p + 1, c, f)         # other parent id
    elif kind == 3:
        tags[l] = (p, c + 1, f)         # other child index
    else:
        tags[l] = (p, c + 2, True)      # a second last child
    frags[i] = (tuple(tags), tok, sc)
    return frags


@pytest.mark.parametrize("depth", [1, 2, 3])
def test_bruteforce_defects(depth):
    rng = random.Random(100 + depth)
    seen = set()
    for n_case, (frags, sizes, po, so, kk) in enumerate(_cases(depth, exhaustive_upto=3, samples=4)):
        if n_case % 3:
            continue
        bad = mutate(frags, rng)
        # new cut over the mutated list
        c = list(cuts(len(bad)))
        sz = rng.choice(c)
        want = evaluate(depth, po, so, kk, bad, sz)
        seen.update(st for st, *_ in want)
        compare(depth, po, so, kk, bad, sz, status_only=True)
    assert ({-4, -5, -6} if depth > 1 else {-4, -5}) <= seen


def test_bruteforce_bad_offsets():
    frags = tree_fragments([2, 3])
    for b in range(3):
        want = [0] * b + [-1] * (3 - b)
        got = [d.status for d in run_oracle(2, [0, 1], [0, 0], [0, 0], frags, [2, 2, 1], corrupt=b)]
        assert got == want
