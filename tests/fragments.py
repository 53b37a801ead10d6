"""Helpers that turn plain fragment lists into batches (test infrastructure).

A fragment is ``(tags, tokens, score)`` where ``tags`` lists
``(parent_id, child_index, last)`` per level, outermost first.
"""
from __future__ import annotations

import numpy as np


def pack(p, c, f):
    return (int(p) << 32) | (int(bool(f)) << 31) | int(c)


def to_batch(frags, depth, with_score):
    n = len(frags)
    tags = np.zeros((depth, n), dtype=np.uint64)
    off = np.zeros(n + 1, dtype=np.uint32)
    toks = []
    for i, (t, tok, _s) in enumerate(frags):
        for l in range(depth):
            tags[l, i] = pack(*t[l])
        off[i + 1] = off[i] + len(tok)
        toks.extend(tok)
    score = np.asarray([s for _t, _tok, s in frags], dtype=np.float32) if with_score else None
    return dict(n=n, tags=tags, off=off, payload=np.asarray(toks, dtype=np.int32), score=score)


def split(frags, batch_sizes):
    out, s = [], 0
    for nb in batch_sizes:
        out.append(frags[s:s + nb])
        s += nb
    return out


def tree_fragments(shape, rng=None, depth=None, id_base=100, score_fn=None, tok_fn=None):
    """Fragments (DFS order) of one source tree.  ``shape`` nests child
    counts: an int is a leaf-parent with that many leaves, a list holds the
    shapes of the children.  Group ids are unique per level."""
    counters = {}

    def new_id(level):
        counters[level] = counters.get(level, 0) + 1
        return id_base * (level + 1) + counters[level]

    out = []

    def walk(node, level, prefix):
        gid = new_id(level)
        if isinstance(node, int):
            for c in range(node):
                tags = prefix + [(gid, c, c == node - 1)]
                out.append(tags)
        else:
            for c, child in enumerate(node):
                walk(child, level + 1, prefix + [(gid, c, c == len(node) - 1)])

    walk(shape, 0, [])
    frags = []
    for k, tags in enumerate(out):
        tok = tok_fn(k) if tok_fn else [1000 * (k + 1) + j for j in range(1 + k % 3)]
        sc = score_fn(k) if score_fn else float(k % 5) - 2.0
        frags.append((tuple(tags), tok, sc))
    return frags


def window_stream(n_groups, n_children, window, batch, seed, topk=False):
    """Depth 2: one source (level 0) with n_groups leaf-parent groups (level
    1) of n_children leaves each, children in a random order; at most
    `window` groups are open at once (a group starts when one ends), the
    leaves of the open ones interleaved at random."""
    from gen.streams import Stream

    rng = np.random.default_rng(seed)
    live, nxt, g_of, c_of = [], 0, [], []
    while nxt < n_groups or live:
        while len(live) < window and nxt < n_groups:
            live.append([nxt, list(rng.permutation(n_children))])
            nxt += 1
        k = int(rng.integers(0, len(live)))
        g_of.append(live[k][0])
        c_of.append(live[k][1].pop(0))
        if not live[k][1]:
            live.pop(k)
    g = np.asarray(g_of, np.uint64)
    c = np.asarray(c_of, np.uint64)
    n = len(g)
    tags = np.zeros((2, n), np.uint64)
    tags[0] = (np.uint64(1) << np.uint64(32)) | ((g == n_groups - 1).astype(np.uint64) << np.uint64(31)) | g
    tags[1] = ((np.uint64(1000) + g) << np.uint64(32)) | ((c == n_children - 1).astype(np.uint64) << np.uint64(31)) | c
    lens = rng.integers(0, 5, size=n)
    off = np.concatenate([[0], np.cumsum(lens)]).astype(np.int64)
    payload = rng.integers(0, 1 << 30, size=int(off[-1])).astype(np.int32)
    score = rng.standard_normal(n).astype(np.float32) if topk else None
    sizes = [batch] * (n // batch) + ([n % batch] if n % batch else [])
    return Stream(name="window", depth=2, payload_op=(0, 1), score_op=(0, 2 if topk else 0),
                  topk_k=(0, 3 if topk else 0), tags=tags, off=off, payload=payload, score=score,
                  batch_sizes=np.asarray(sizes), meta={})
