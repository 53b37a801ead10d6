"""Seeded synthetic fragment streams shaped like the paper's workloads.

This module only produces inputs: ancestry tags, payload spans and scores in
arrival order, cut into batches.  It holds none of the aggregation
arithmetic, and both the CPU oracle harness and the CUDA path read the same
streams from here.
"""
from .streams import (  # noqa: F401
    CONCAT, NONE, S_MAX, S_NONE, S_TOPK, TOKEN_VOCAB, Stream, CONFIG_NAMES,
    make_stream, pack_tags, stream_from_leaves, SplitInput, make_split_input,
)
