"""Routing by ancestry -- TEST INFRASTRUCTURE ONLY.

Same rules as the rest of ``oracle/``: only ``tests/``,
``__graft_entry__.smoke()`` and the benchmark's CPU legs may use it, and it
shares no code with the CUDA library.

What it follows (Sec. 4.3): the aggregation at a pmap exit needs every element
of a group at the same physical instance of the next stage, so all elements
with the same ancestry tags are routed to the same instance -- like ECMP, but
keyed on the tags -- and the instance that a new "flow" of tags goes to may be
chosen by load rather than by a hash.  Sec. 5: the controller picks replicas
by these rules and by watching queue lengths.

Readings (the paper gives no more detail):

* A flow is the group at the routing level L: the fragments whose tags agree
  on levels 0..L.  Parent ids are unique per level, so the pair (L, p_L) names
  the flow.
* HASH: replica = splitmix64(L << 32 | p_L) mod R, with the splitmix64
  finaliser (Steele, Lea, Flood, "Fast splittable pseudorandom number
  generators", 2014).
* LEAST_LOADED: a flow already placed keeps its replica.  The new flows of a
  batch, in the order of their first fragment, are dealt round-robin over the
  replicas ordered by load at the start of the batch (fewest first, ties to
  the lower index).  Without a queue-length signal from the instances, a
  replica's load is the number of fragments routed to it so far.
* A flow is forgotten when the aggregator reports its group complete (a
  record at level L with its parent id); a later fragment of the same id is
  then a new flow.
* The batch is partitioned stably: replica r's sub-batch holds its fragments
  in arrival order, as a batch of its own (level-major tags, payload offsets
  from 0, payload, scores).
"""
from __future__ import annotations

import numpy as np

HASH, LEAST_LOADED = 0, 1
_M64 = (1 << 64) - 1


def splitmix64_mix(x: int) -> int:
    """The splitmix64 output function (finaliser) of a 64-bit state."""
    x &= _M64
    x = ((x ^ (x >> 30)) * 0xBF58476D1CE4E5B9) & _M64
    x = ((x ^ (x >> 27)) * 0x94D049BB133111EB) & _M64
    return x ^ (x >> 31)


class RouterOracle:
    def __init__(self, depth, level, n_replicas, policy):
        assert 0 <= level < depth and n_replicas >= 1 and policy in (HASH, LEAST_LOADED)
        self.depth, self.level, self.R, self.policy = depth, level, n_replicas, policy
        self.flows = {}                  # parent id at the routing level -> replica
        self.load = [0] * n_replicas     # fragments routed to each replica

    def replica_of_flows(self, pids):
        """Replica of each fragment's flow, in arrival order (updates the state)."""
        if self.policy == HASH:
            return [splitmix64_mix((self.level << 32) | int(p)) % self.R for p in pids]
        order = sorted(range(self.R), key=lambda r: (self.load[r], r))
        k = 0
        out = []
        for p in pids:
            p = int(p)
            if p not in self.flows:
                self.flows[p] = order[k % self.R]
                k += 1
            out.append(self.flows[p])
        return out

    def route(self, batch):
        """batch: dict(n, tags [D, n] uint64, off [n+1], payload, score or None).

        Returns (replica [n], perm [n], counts [R + 1], parts) where perm lists
        the fragments grouped by replica in arrival order, counts[r] is where
        replica r's fragments start in perm, and parts[r] is replica r's
        sub-batch (a dict like the input)."""
        n = batch["n"]
        tags = np.asarray(batch["tags"], dtype=np.uint64).reshape(self.depth, n)
        pids = (tags[self.level] >> np.uint64(32)).tolist()
        replica = np.asarray(self.replica_of_flows(pids), dtype=np.int64)
        for r in replica.tolist():
            self.load[r] += 1
        perm = np.argsort(replica, kind="stable")
        counts = np.zeros(self.R + 1, dtype=np.int64)
        np.add.at(counts, replica + 1, 1)
        counts = np.cumsum(counts)
        off = np.asarray(batch["off"], dtype=np.int64)
        parts = []
        for r in range(self.R):
            idx = perm[counts[r]:counts[r + 1]]
            lens = off[idx + 1] - off[idx]
            sub_off = np.concatenate([[0], np.cumsum(lens)]).astype(np.int64)
            pay = (np.concatenate([batch["payload"][off[i]:off[i + 1]] for i in idx])
                   if len(idx) else np.zeros(0, np.int32)).astype(np.int32)
            parts.append(dict(n=len(idx), tags=np.ascontiguousarray(tags[:, idx]), off=sub_off,
                              payload=pay,
                              score=None if batch["score"] is None else np.asarray(batch["score"])[idx]))
        return replica, perm, counts, parts

    def release(self, records):
        """Forget the flows whose groups the aggregator reported complete."""
        for r in records:
            if int(r["level"]) == self.level:
                self.flows.pop(int(r["parent_id"]), None)
