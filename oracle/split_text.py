"""split_text definition -- TEST INFRASTRUCTURE ONLY.

Same rules as the rest of ``oracle/``: only ``tests/``,
``__graft_entry__.smoke()`` and the benchmark's CPU legs may use it, and it
shares no code with the CUDA library.

What it follows:

* Sec. 3.1 (hierarchical datatypes) and Sec. 3.2 (data manipulation
  operators): ``split_text`` turns one text item of a ``Delimiter`` type into
  a stream of smaller ``Delimiter`` items (a line into words, a paragraph
  into lines), one level of hierarchy below the item.
* Sec. 4.2 (nested ancestry): at the pmap entry every child keeps its
  parent's tags and gets one new tag: the parent's id at the new level, the
  child's index in the parent's stream, and the end-of-output delimiter (the
  last flag) on the final child (Sec. 3.1).

Readings where the paper says nothing: a delimiter token ends the piece it
closes and stays in it; an item that ends with a delimiter has no trailing
empty piece; an empty item has one empty piece.  The pieces therefore tile
the item: concatenated in order, they give it back.
"""
from __future__ import annotations

import numpy as np


def _pack(pid, child, last):
    return ((np.asarray(pid, dtype=np.uint64) << np.uint64(32))
            | (np.asarray(last, dtype=np.uint64) << np.uint64(31))
            | np.asarray(child, dtype=np.uint64))


def split_pieces(tokens, a, b, delims):
    """Exclusive end positions of the pieces of tokens[a:b]."""
    ends = (np.flatnonzero(np.isin(tokens[a:b], np.asarray(list(delims), dtype=np.int64))) + a + 1).tolist()
    if not ends or ends[-1] != b:
        ends.append(b)  # the piece after the last delimiter; an empty item's only piece
    return ends


def split_text(src_tags, src_id, tok_off, tokens, delims):
    """src_tags: uint64 [depth_in, n_src] (level-major, may have depth_in = 0),
    src_id: uint32 [n_src], tok_off: [n_src + 1] offsets into tokens, tokens:
    int32, delims: delimiter token ids.

    Returns (tags, off): tags uint64 [depth_in + 1, n_frag] level-major, off
    int64 [n_frag + 1] offsets of the pieces into ``tokens``, pieces in stream
    order, each stream's pieces in position order."""
    src_tags = np.asarray(src_tags, dtype=np.uint64).reshape(-1, len(src_id))
    depth_in = src_tags.shape[0]
    tokens = np.asarray(tokens)
    ends, src_of, kidx, last = [], [], [], []
    for s in range(len(src_id)):
        e = split_pieces(tokens, int(tok_off[s]), int(tok_off[s + 1]), delims)
        ends += e
        src_of += [s] * len(e)
        kidx += list(range(len(e)))
        last += [False] * (len(e) - 1) + [True]
    src_of = np.asarray(src_of, dtype=np.int64)
    tags = np.empty((depth_in + 1, len(ends)), dtype=np.uint64)
    for l in range(depth_in):
        tags[l] = src_tags[l][src_of]
    tags[depth_in] = _pack(np.asarray(src_id, dtype=np.uint64)[src_of], kidx, last)
    off = np.asarray([int(tok_off[0])] + ends, dtype=np.int64)
    return tags, off
