"""GB300-native re-aggregation of streamed fragments by nested ancestry.

The hot path (Alto, arxiv 2403.04311, Sec. 3.1-4.3) is a CUDA library for
sm_103a behind a four-call C ABI (``include/alto_agg.h``); this package builds
it in-tree and binds it with ctypes.  There is no CPU implementation here.
"""
from ._binding import (  # noqa: F401
    EXPORTS, OK, EINVAL, ENOMEM, ENOSPC, EDUP, ELAST, EINCONSIST, ECLOSED, ETIMEOUT, ECUDA,
    STATUS_NAMES, PAYLOAD_NONE, PAYLOAD_CONCAT, SCORE_NONE, SCORE_MAX, SCORE_TOPK, FLAG_STREAM_RELEASE, FLAG_DOUBLE_RING, OPS_PARTIAL,
    RECORD_DTYPE, PAIR_DTYPE, Aggregator, Drain, alto_agg_config, alto_allocator, alto_batch,
    alto_drain, alto_agg_create, alto_agg_push_batch, alto_agg_drain, alto_agg_stats,
    alto_agg_destroy, alto_agg_profile, alto_agg_profile_read, alto_agg_oneshot_noalloc,
    load_library, make_config, alto_split_args, alto_split_scratch_bytes, alto_split_text, split_text,
    Router, ROUTE_HASH, ROUTE_LEAST_LOADED,
    STAGE_NAMES, PROFILE_OFF, PROFILE_STAGES, PROFILE_HOT,
)
from ._build import build  # noqa: F401
from .device_batches import DeviceBatch, to_device  # noqa: F401
