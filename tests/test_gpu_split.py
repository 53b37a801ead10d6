"""split_text on the GPU against the oracle, bit for bit, through the C ABI.

Tags and piece offsets must be identical; the cases span several scan tiles
(4,096 elements a tile) and a ragged tail, empty streams, streams ending with a
delimiter, runs of delimiters, one stream much longer than the rest, zero to
two levels of input tags, and the 100M-token full-size input.  The pipeline
test pushes the GPU's pieces into the GPU aggregator with CONCAT at the new
level and compares the drain with the oracle's split + aggregation.
"""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

import oracle
import paper_2403_04311_gb300 as alto
from gen import make_split_input
from gpu_harness import assert_same, run_gpu_batches, run_oracle_batches

pytestmark = pytest.mark.gpu


def gpu_split(src_tags, src_id, tok_off, tokens, delims, cap=None, misalign=False):
    st_t = None if src_tags.shape[0] == 0 else torch.as_tensor(src_tags.view(np.int64), device="cuda")
    sid = torch.as_tensor(np.asarray(src_id, dtype=np.uint32).view(np.int32), device="cuda")
    off = torch.as_tensor(np.asarray(tok_off, dtype=np.uint32).view(np.int32), device="cuda")
    tok = torch.as_tensor(np.asarray(tokens, dtype=np.int32), device="cuda")
    if misalign:
        # the same tokens one element into a larger buffer: 4-byte but not
        # 16-byte aligned, so every token is read on its own
        buf = torch.zeros(tok.numel() + 1, dtype=torch.int32, device="cuda")
        buf[1:] = tok
        tok = buf[1:]
    st, n, tags, poff = alto.split_text(st_t, sid, off, tok, list(delims), cap_frag=cap)
    if st != alto.OK:
        return st, n, None, None
    return st, n, tags.cpu().numpy().view(np.uint64), poff.cpu().numpy().view(np.uint32).astype(np.int64)


def _random_case(rng, n_src, max_len, delims, depth_in, long_one=False):
    lens = rng.integers(0, max_len + 1, size=n_src)
    if long_one:
        lens[rng.integers(0, n_src)] = 50_000
    lens[rng.random(n_src) < 0.1] = 0
    toks = rng.integers(0, 40, size=int(lens.sum())).astype(np.int32)
    # some streams end with a delimiter, some hold runs of them
    off = np.concatenate([[0], np.cumsum(lens)]).astype(np.int64)
    for s in range(n_src):
        if lens[s] and rng.random() < 0.3:
            toks[off[s + 1] - 1] = delims[0]
        if lens[s] > 3 and rng.random() < 0.2:
            toks[off[s]:off[s] + 3] = delims[-1]
    src_tags = rng.integers(0, 2**63, size=(depth_in, n_src), dtype=np.uint64)
    src_id = (rng.permutation(10 * n_src) + 1)[:n_src].astype(np.uint32)
    return src_tags, src_id, off, toks


@pytest.mark.parametrize("n_src,max_len,depth_in,long_one", [
    (1, 0, 0, False), (1, 5, 1, False), (7, 30, 2, False), (300, 60, 1, False),
    (2000, 40, 0, True), (5000, 9, 2, False)])
def test_split_matches_oracle(n_src, max_len, depth_in, long_one):
    rng = np.random.default_rng(n_src + max_len)
    delims = [3, 7, 11]
    src_tags, src_id, off, toks = _random_case(rng, n_src, max_len, delims, depth_in, long_one)
    want_tags, want_off = oracle.split_text(src_tags, src_id, off, toks, delims)
    st, n, tags, poff = gpu_split(src_tags, src_id, off, toks, delims)
    assert st == alto.OK
    assert n == want_tags.shape[1]
    assert np.array_equal(tags, want_tags)
    assert np.array_equal(poff, want_off)


@pytest.mark.parametrize("n_src,max_len", [(7, 30), (2000, 40)])
def test_split_unaligned_tokens(n_src, max_len):
    rng = np.random.default_rng(n_src + 1)
    delims = [3, 7, 11]
    src_tags, src_id, off, toks = _random_case(rng, n_src, max_len, delims, 1, n_src > 100)
    want_tags, want_off = oracle.split_text(src_tags, src_id, off, toks, delims)
    st, n, tags, poff = gpu_split(src_tags, src_id, off, toks, delims, misalign=True)
    assert st == alto.OK and n == want_tags.shape[1]
    assert np.array_equal(tags, want_tags)
    assert np.array_equal(poff, want_off)


def test_split_errors():
    src_tags = np.zeros((0, 2), np.uint64)
    toks = np.asarray([1, 3, 2, 3], np.int32)
    st, n, _, _ = gpu_split(src_tags, [5, 6], [0, 2, 4], toks, [3], cap=1)
    assert st == alto.ENOSPC and n == 2
    st, n, _, _ = gpu_split(src_tags, [5, 6], [0, 3, 2], toks, [3])    # decreasing offsets
    assert st == alto.EINVAL
    st, n, _, _ = gpu_split(src_tags, [5, 6], [0, 2, 3], toks, [3])    # does not end at n_tokens
    assert st == alto.EINVAL


def test_split_then_aggregate_matches_oracle():
    """Pieces straight from the GPU split into the GPU aggregator (CONCAT at the
    new level), against the oracle's split + aggregation."""
    si = make_split_input(n_streams=300, tokens_per_stream=700, empty_every=13)
    st, n, tags, poff = gpu_split(si.src_tags, si.src_id, si.tok_off, si.tokens, si.delims)
    assert st == alto.OK
    otags, ooff = oracle.split_text(si.src_tags, si.src_id, si.tok_off, si.tokens, si.delims)
    batch = dict(n=n, tags=np.ascontiguousarray(tags), off=poff.astype(np.uint32), payload=si.tokens,
                 score=None)
    obatch = dict(n=n, tags=otags, off=ooff.astype(np.uint32), payload=si.tokens, score=None)
    caps = dict(max_batch_fragments=n, max_batch_payload=len(si.tokens), max_open_groups=4096,
                arena_elems=1 << 20, out_records=n + 1024, out_payload_elems=len(si.tokens) + 16,
                out_topk=16, max_emit_children=2 * n)
    _, g = run_gpu_batches(2, [0, 1], [0, 0], [0, 0], [batch], caps)
    o = run_oracle_batches(2, [0, 1], [0, 0], [0, 0], [obatch])
    assert_same(o, g, "split+aggregate")
    # and every stream came back whole
    _st, rec, pay, _ = g[0]
    streams = {int(r["parent_id"]): pay[int(r["payload_off"]):int(r["payload_off"]) + int(r["payload_len"])]
               for r in rec[rec["level"] == 1]}
    for s in range(len(si.src_id)):
        assert np.array_equal(streams[int(si.src_id[s])], si.tokens[si.tok_off[s]:si.tok_off[s + 1]])


@pytest.mark.slow
def test_split_fullsize():
    """4,096 streams x 24,414 tokens (100M tokens), sentences of U{1..64}."""
    si = make_split_input()
    want_tags, want_off = oracle.split_text(si.src_tags, si.src_id, si.tok_off, si.tokens, si.delims)
    st, n, tags, poff = gpu_split(si.src_tags, si.src_id, si.tok_off, si.tokens, si.delims)
    assert st == alto.OK and n == want_tags.shape[1]
    assert np.array_equal(tags, want_tags)
    assert np.array_equal(poff, want_off)
