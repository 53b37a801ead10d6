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
