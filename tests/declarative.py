"""Non-incremental evaluation of the aggregation definition, for tiny inputs.

Test infrastructure: it shares no code with the oracle (``oracle/``) nor with
the CUDA library.  Where the oracle walks fragments in arrival order and keeps
running counts, this module rebuilds the whole ancestry tree for every batch
prefix and evaluates the recursive completion predicate from scratch
(Sec. 3.1: a stream is complete once its end-of-output delimiter has arrived
and, Sec. 4.2, every nested level below it is complete).  A group is emitted in
the batch whose prefix first makes it complete; its completion sequence number
is the smallest arrival index whose prefix makes it complete, found by trying
every prefix.  Records are ordered by (completion seq, deeper level first).

With streaming release (Sec. 3.2: the reordered outputs of a pmap flow on as
a stream), after each batch every open group at the CONCAT level whose run of
complete children 0..r-1 is longer than the run it already released gets a
partial record for the new children (ops bit 0x80, n_children = r, seq = the
latest completion seq among them, no score); a group's final record then
carries only the children it had not released.

Fragments are plain Python: ``(tags, tokens, score)`` with ``tags`` a tuple of
``(parent_id, child_index, last)`` per level, outermost first.
"""
from __future__ import annotations

import math
import struct

OK, EINVAL, EDUP, ELAST, EINCONSIST, ECLOSED = 0, -1, -4, -5, -6, -7
_PRIORITY = {EINVAL: 5, EDUP: 4, EINCONSIST: 3, ELAST: 2, ECLOSED: 1, OK: 0}


def order_key(x: float) -> int:
    """Integer whose natural order is IEEE-754 totalOrder on float32."""
    (u,) = struct.unpack("<I", struct.pack("<f", x))
    return (u ^ 0xFFFFFFFF) if u & 0x80000000 else (u | 0x80000000)


class _Tree:
    def __init__(self, depth, frags):
        self.depth = depth
        self.kids = {}      # (l, p) -> {c: child id (l < D-1) or fragment index}
        self.flagged = {}   # (l, p) -> set of flagged child indices
        for i, (tags, _tok, _s) in enumerate(frags):
            for l, (p, c, f) in enumerate(tags):
                g = (l, p)
                self.kids.setdefault(g, {})
                self.flagged.setdefault(g, set())
                self.kids[g][c] = tags[l + 1][0] if l < depth - 1 else i
                if f:
                    self.flagged[g].add(c)

    def last(self, g):
        fl = self.flagged.get(g, set())
        return min(fl) if len(fl) == 1 else None

    def complete(self, g):
        last = self.last(g)
        if last is None:
            return False
        ch = self.kids[g]
        if set(ch) != set(range(last + 1)):
            return False
        l, _ = g
        if l == self.depth - 1:
            return True
        return all(self.complete((l + 1, ch[c])) for c in range(last + 1))

    def leaves(self, g):
        """Fragment indices of the subtree, in child-index path order."""
        l, _ = g
        ch = self.kids[g]
        out = []
        for c in sorted(ch):
            if l == self.depth - 1:
                out.append(ch[c])
            else:
                out.extend(self.leaves((l + 1, ch[c])))
        return out


def violations(depth, frags):
    """Error classes that the fragment set violates (ECLOSED excluded)."""
    v = set()
    leaf_slots = {}
    up = {}
    slot_child = {}
    flagged = {}
    maxc = {}
    for tags, _tok, _s in frags:
        lp, lc, _ = tags[depth - 1]
        leaf_slots[(lp, lc)] = leaf_slots.get((lp, lc), 0) + 1
        for l, (p, c, f) in enumerate(tags):
            g = (l, p)
            if l > 0:
                up.setdefault(g, set()).add(tags[l - 1])
            if l < depth - 1:
                slot_child.setdefault((l, p, c), set()).add(tags[l + 1][0])
            if f:
                flagged.setdefault(g, set()).add(c)
            maxc[g] = max(maxc.get(g, -1), c)
    if any(n > 1 for n in leaf_slots.values()):
        v.add(EDUP)
    if any(len(s) > 1 for s in up.values()) or any(len(s) > 1 for s in slot_child.values()):
        v.add(EINCONSIST)
    for g, fl in flagged.items():
        if len(fl) > 1 or maxc[g] > min(fl):
            v.add(ELAST)
    return v


def _closed(depth, frags, upto):
    """True if some fragment among frags[:upto] references a group that was
    already complete in the prefix strictly before it."""
    for x in range(upto):
        t = _Tree(depth, frags[:x])
        for l, (p, _c, _f) in enumerate(frags[x][0]):
            if (l, p) in t.kids and t.complete((l, p)):
                return True
    return False


def _completion_seq(depth, frags, end, g):
    """Smallest arrival index whose prefix makes group g complete."""
    return next(x for x in range(end) if g in _Tree(depth, frags[:x + 1]).kids
                and _Tree(depth, frags[:x + 1]).complete(g))


def evaluate(depth, payload_op, score_op, topk_k, frags, batch_sizes, csr_ok=None, stream_release=False):
    """Per batch: (status, records, payload, topk).  After the first batch
    with an error every later batch reports the same status and nothing else.
    ``csr_ok[b] = False`` marks a batch whose offsets or scores are invalid.
    Records are dicts with the record fields; payload offsets are relative to
    the batch's own payload list."""
    out = []
    status = OK
    start = 0
    prev_complete = set()
    released = {}                 # CONCAT-level group -> children released so far
    cl = payload_op.index(1) if 1 in list(payload_op)[:depth] else None
    for b, nb in enumerate(batch_sizes):
        end = start + nb
        if status != OK:
            out.append((status, [], [], []))
            start = end
            continue
        errs = set()
        if csr_ok is not None and not csr_ok[b]:
            errs.add(EINVAL)
        else:
            errs |= violations(depth, frags[:end])
            if _closed(depth, frags, end):
                errs.add(ECLOSED)
        if errs:
            status = max(errs, key=lambda e: _PRIORITY[e])
            out.append((status, [], [], []))
            start = end
            continue
        tree = _Tree(depth, frags[:end])
        now = {g for g in tree.kids if tree.complete(g)}
        new = now - prev_complete
        prev_complete = now
        recs = []
        for g in new:
            recs.append((_completion_seq(depth, frags, end, g), -g[0], g, None))
        if stream_release and cl is not None:
            for g in tree.kids:
                if g[0] != cl or g in now:
                    continue
                r, seqs = 0, []
                while r in tree.kids[g]:
                    if cl == depth - 1:
                        seqs.append(tree.kids[g][r])
                    else:
                        child = (cl + 1, tree.kids[g][r])
                        if not tree.complete(child):
                            break
                        seqs.append(_completion_seq(depth, frags, end, child))
                    r += 1
                r0 = released.get(g, 0)
                if r > r0:
                    recs.append((max(seqs[r0:r]), -cl, g, (r0, r)))
                    released[g] = r
        recs.sort()
        payload, topk, records = [], [], []
        for s, _, g, part in recs:
            l, p = g
            if part is not None:          # partial record: children part[0]..part[1]-1
                rec = dict(completion_seq=s, parent_id=p, n_children=part[1], level=l, ops=1 | 0x80,
                           payload_off=len(payload), topk_off=len(topk), topk_n=0, score=0.0)
                for c in range(part[0], part[1]):
                    sub = [tree.kids[g][c]] if l == depth - 1 else tree.leaves((l + 1, tree.kids[g][c]))
                    for i in sub:
                        payload.extend(frags[i][1])
                rec["payload_len"] = len(payload) - rec["payload_off"]
                records.append(rec)
                continue
            last = tree.last(g)
            leaves = tree.leaves(g)
            if stream_release and l == cl and released.get(g, 0):
                skip = set()
                for c in range(released[g]):
                    skip.update([tree.kids[g][c]] if l == depth - 1 else tree.leaves((l + 1, tree.kids[g][c])))
                payload_leaves = [i for i in leaves if i not in skip]
            else:
                payload_leaves = leaves
            rec = dict(completion_seq=s, parent_id=p, n_children=last + 1, level=l,
                       ops=payload_op[l] | (score_op[l] << 2), payload_off=len(payload),
                       topk_off=len(topk), topk_n=0, score=0.0)
            if payload_op[l] == 1:
                for i in payload_leaves:
                    payload.extend(frags[i][1])
            rec["payload_len"] = len(payload) - rec["payload_off"]
            if score_op[l] != 0:
                rec["score"] = max((frags[i][2] for i in leaves), key=order_key)
            if score_op[l] == 2:
                kids = []
                for c in range(last + 1):
                    if l == depth - 1:
                        sc = frags[tree.kids[g][c]][2]
                    else:
                        sub = tree.leaves((l + 1, tree.kids[g][c]))
                        sc = max((frags[i][2] for i in sub), key=order_key)
                    kids.append((c, sc))
                kids.sort(key=lambda cs: (-order_key(cs[1]), cs[0]))
                sel = kids[:topk_k[l]]
                topk.extend(sel)
                rec["topk_n"] = len(sel)
            records.append(rec)
        out.append((OK, records, payload, topk))
        start = end
    return out


def same_float(a: float, b: float) -> bool:
    """Bit-identical float32 values."""
    if math.isnan(a) or math.isnan(b):
        return False
    return struct.pack("<f", a) == struct.pack("<f", b)
