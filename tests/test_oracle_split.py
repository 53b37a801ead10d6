"""The split_text oracle against definitions it does not share code with.

* newline splitting = ``str.splitlines(keepends=True)`` on texts whose only
  line break is ``\\n`` (Python's own routine; non-empty texts);
* several delimiters = a regular expression that takes a run of
  non-delimiters with the delimiter that closes it, or the final run;
* invariants: the pieces tile each stream, every piece but a stream's last
  ends with a delimiter and holds no other, child indices count up from 0,
  the last flag is on the final piece only, the stream's own tags are copied;
* special cases: an empty stream has one empty piece, a stream ending with a
  delimiter has no trailing empty piece, consecutive delimiters are pieces of
  their own;
* round trip through the aggregation oracle: split, then CONCAT at the new
  level, gives every stream back (Sec. 3.2: the stream is reconstituted).
"""
import random
import re

import numpy as np

import oracle


def _pack(p, c, f):
    return (int(p) << 32) | (int(bool(f)) << 31) | int(c)


def _streams(texts):
    toks = np.asarray([ord(ch) for t in texts for ch in t], dtype=np.int32)
    off = np.concatenate([[0], np.cumsum([len(t) for t in texts])]).astype(np.int64)
    return toks, off


def _pieces_as_text(tags, off, toks, depth_in):
    out = {}
    pid = (tags[depth_in] >> np.uint64(32)).astype(np.int64)
    for f in range(len(pid)):
        out.setdefault(int(pid[f]), []).append("".join(chr(x) for x in toks[off[f]:off[f + 1]]))
    return out


def test_newlines_match_splitlines():
    rng = random.Random(1)
    for _ in range(300):
        texts = ["".join(rng.choice("ab \n") for _ in range(rng.randint(1, 30))) for _ in range(rng.randint(1, 6))]
        toks, off = _streams(texts)
        ids = list(range(100, 100 + len(texts)))
        tags, poff = oracle.split_text(np.zeros((0, len(texts)), np.uint64), ids, off, toks, [ord("\n")])
        got = _pieces_as_text(tags, poff, toks, 0)
        for i, t in enumerate(texts):
            assert got[ids[i]] == t.splitlines(keepends=True), t


def test_several_delimiters_match_regex():
    rng = random.Random(2)
    pat = re.compile(r"[^ \n.]*[ \n.]|[^ \n.]+$")
    for _ in range(300):
        t = "".join(rng.choice("ab. \n") for _ in range(rng.randint(1, 40)))
        toks, off = _streams([t])
        tags, poff = oracle.split_text(np.zeros((0, 1), np.uint64), [5], off, toks, [ord(" "), ord("\n"), ord(".")])
        assert _pieces_as_text(tags, poff, toks, 0)[5] == pat.findall(t), t


def test_invariants_and_special_cases():
    rng = np.random.default_rng(3)
    delims = [7, 9]
    for trial in range(200):
        n_src = int(rng.integers(1, 8))
        lens = rng.integers(0, 12, size=n_src)
        toks = rng.integers(0, 12, size=int(lens.sum())).astype(np.int32)
        off = np.concatenate([[0], np.cumsum(lens)]).astype(np.int64)
        depth_in = int(rng.integers(0, 3))
        src_tags = rng.integers(0, 2**63, size=(depth_in, n_src), dtype=np.uint64)
        ids = rng.permutation(1000)[:n_src] + 1
        tags, poff = oracle.split_text(src_tags, ids, off, toks, delims)
        n_frag = tags.shape[1]
        assert poff[0] == 0 and poff[-1] == off[-1] and np.all(np.diff(poff) >= 0)
        pid = (tags[depth_in] >> np.uint64(32)).astype(np.int64)
        cid = (tags[depth_in] & np.uint64(0x7FFFFFFF)).astype(np.int64)
        lst = ((tags[depth_in] >> np.uint64(31)) & np.uint64(1)).astype(bool)
        f = 0
        for s in range(n_src):
            a, b = int(off[s]), int(off[s + 1])
            pieces = []
            k = 0
            while f < n_frag and pid[f] == ids[s] and (k == 0 or not lst[f - 1]):
                assert cid[f] == k
                for l in range(depth_in):
                    assert tags[l, f] == src_tags[l, s]
                pieces.append(toks[poff[f]:poff[f + 1]])
                f += 1
                k += 1
            assert lst[f - 1] and not lst[f - k:f - 1].any()
            # tiling and delimiter placement
            assert np.array_equal(np.concatenate(pieces) if pieces else np.zeros(0, np.int32), toks[a:b])
            for p in pieces[:-1]:
                assert len(p) >= 1 and p[-1] in delims and not np.isin(p[:-1], delims).any()
            assert not np.isin(pieces[-1][:-1], delims).any()
            if a == b:
                assert len(pieces) == 1 and len(pieces[0]) == 0
            elif toks[b - 1] in delims:
                assert len(pieces[-1]) >= 1 and pieces[-1][-1] in delims
            n_delim = int(np.isin(toks[a:b], delims).sum())
            want = n_delim + (0 if (b > a and toks[b - 1] in delims) else 1)
            assert len(pieces) == want
        assert f == n_frag


def test_consecutive_delimiters_are_pieces():
    toks = np.asarray([1, 9, 9, 9, 2], dtype=np.int32)
    tags, poff = oracle.split_text(np.zeros((0, 1), np.uint64), [3], [0, 5], toks, [9])
    assert poff.tolist() == [0, 2, 3, 4, 5]
    assert tags[0].tolist() == [_pack(3, 0, 0), _pack(3, 1, 0), _pack(3, 2, 0), _pack(3, 3, 1)]


def test_round_trip_through_concat():
    """Split streams that are children of one root, aggregate with CONCAT at
    the new level: every stream comes back, in order."""
    rng = np.random.default_rng(4)
    n_src = 40
    lens = rng.integers(0, 30, size=n_src)
    toks = rng.integers(0, 6, size=int(lens.sum())).astype(np.int32)
    off = np.concatenate([[0], np.cumsum(lens)]).astype(np.int64)
    src_tags = np.asarray([[_pack(77, s, s == n_src - 1) for s in range(n_src)]], dtype=np.uint64)
    ids = np.arange(500, 500 + n_src)
    tags, poff = oracle.split_text(src_tags, ids, off, toks, [0, 3])
    n = tags.shape[1]
    perm = rng.permutation(n)            # arrival order unrelated to stream order
    batch = dict(n=n, tags=np.ascontiguousarray(tags[:, perm]),
                 off=np.concatenate([[0], np.cumsum((poff[1:] - poff[:-1])[perm])]).astype(np.uint32),
                 payload=np.concatenate([toks[poff[i]:poff[i + 1]] for i in perm]).astype(np.int32)
                 if n else np.zeros(0, np.int32),
                 score=None)
    o = oracle.Oracle(2, [0, 1], [0, 0], [0, 0])
    o.push_batch(batch)
    d = o.drain()
    o.close()
    assert d.status == 0
    recs = d.records
    got = {}
    for r in recs[recs["level"] == 1]:
        got[int(r["parent_id"])] = d.payload[int(r["payload_off"]):int(r["payload_off"]) + int(r["payload_len"])]
    assert len(got) == n_src
    for s in range(n_src):
        assert np.array_equal(got[int(ids[s])], toks[off[s]:off[s + 1]])
