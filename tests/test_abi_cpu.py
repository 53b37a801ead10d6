"""C-ABI library: builds for sm_103a, loads, exports every declared entry
point, and its host-side argument checks answer without touching a GPU."""
import ctypes
import os
import re

import pytest

import paper_2403_04311_gb300 as alto

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def declared_functions():
    names = []
    inc = os.path.join(ROOT, "include")
    for f in sorted(os.listdir(inc)):
        if f.endswith(".h"):
            txt = open(os.path.join(inc, f)).read()
            names += re.findall(r"^(?:alto_status|int64_t)\s+(alto_\w+)\s*\(", txt, flags=re.M)
    return names


def test_library_builds_and_exports_every_declared_symbol():
    lib = alto.load_library()
    names = declared_functions()
    assert set(alto.EXPORTS) <= set(names)
    for n in names:
        assert hasattr(lib, n), n


def test_library_is_built_for_sm_103a():
    """Every translation unit is compiled for sm_103a alone (one -gencode,
    no PTX for other targets) and linked into the in-tree library."""
    from paper_2403_04311_gb300 import _build
    assert _build.ARCH == ["-gencode", "arch=compute_103a,code=sm_103a"]
    assert os.path.dirname(_build.LIB) == os.path.join(ROOT, "paper_2403_04311_gb300")
    assert os.path.exists(alto.build())


def _cfg(**kw):
    base = dict(depth=2, payload_op=[0, 1], score_op=[0, 0], max_batch_fragments=1024,
                max_batch_payload=4096)
    base.update(kw)
    d = base.pop("depth")
    return alto.make_config(d, base.pop("payload_op"), base.pop("score_op"), base.pop("topk_k", None), **base)


@pytest.mark.parametrize("bad", [
    dict(depth=0, payload_op=[], score_op=[]),
    dict(depth=9, payload_op=[0] * 9, score_op=[0] * 9),
    dict(payload_op=[1, 1]),                         # two CONCAT levels
    dict(payload_op=[0, 2]),                         # unknown payload op
    dict(score_op=[3, 0]),                           # unknown score op
    dict(score_op=[2, 0], topk_k=[0, 0]),            # TOPK without k
    dict(score_op=[2, 0], topk_k=[33, 0]),           # k above 32
    dict(max_batch_fragments=0),
    dict(max_batch_fragments=1 << 30),
    dict(max_batch_payload=-1),
    dict(max_open_groups=(1 << 25) + 1),
    dict(arena_elems=1 << 32),
    dict(payload_op=[0, 0], stream_release=True),    # streaming release without CONCAT
    dict(flags=16),                                  # unknown flag
])
def test_create_rejects_bad_configs_on_host(bad):
    lib = alto.load_library()
    bad = dict(bad)
    flags = bad.pop("flags", None)
    cfg = _cfg(**bad)
    if flags is not None:
        cfg.flags = flags
    h = ctypes.c_void_p(12345)
    st = lib.alto_agg_create(ctypes.byref(cfg), None, None, ctypes.byref(h))
    assert st == alto.EINVAL
    assert h.value == 12345  # untouched


@pytest.mark.parametrize("flag", ["stream_release", "double_ring", "test_stall", "direct_launch"])
def test_noalloc_refuses_handle_flags_on_host(flag):
    """One batch has nothing to release in a stream and writes the caller's
    buffers, not rings, and the wait-stall test hook is for handles only:
    every flag is refused before any device work."""
    cfg = _cfg(**{flag: True})
    b = alto.alto_batch()
    b.depth = 2
    counts = (ctypes.c_int64 * 4)()
    st = alto.alto_agg_oneshot_noalloc(cfg, b, 0, 0, 0, 0, 0, 0, ctypes.addressof(counts), 0)
    assert st == alto.EINVAL


def test_null_arguments():
    lib = alto.load_library()
    assert lib.alto_agg_destroy(None) == alto.OK
    assert lib.alto_agg_push_batch(None, None, None) == alto.EINVAL
    assert lib.alto_agg_drain(None, None, None) == alto.EINVAL
    assert lib.alto_agg_create(None, None, None, None) == alto.EINVAL
    h = ctypes.c_void_p()
    assert lib.alto_agg_create(ctypes.byref(_cfg()), None, None, None) == alto.EINVAL
    bad_alloc = alto.alto_allocator()
    assert lib.alto_agg_create(ctypes.byref(_cfg()), ctypes.byref(bad_alloc), None,
                               ctypes.byref(h)) == alto.EINVAL


def test_status_codes_match_oracle_and_header():
    import oracle
    txt = open(os.path.join(ROOT, "include", "alto_agg.h")).read()
    vals = dict(re.findall(r"#define ALTO_(E\w+|OK)\s+\(?(-?\d+)\)?", txt))
    assert int(vals["OK"]) == alto.OK == oracle.OK
    for name in ["EINVAL", "ENOMEM", "ENOSPC", "EDUP", "ELAST", "EINCONSIST", "ECLOSED"]:
        assert int(vals[name]) == getattr(alto, name) == getattr(oracle, name)
    assert alto.RECORD_DTYPE == oracle.RECORD_DTYPE


def test_struct_layouts_match_the_header(tmp_path):
    """Every ctypes structure of the binding, and the record and pair dtypes,
    have the size and field offsets that a C compiler gives the header's
    structs (so the binding cannot drift from include/alto_agg.h)."""
    import shutil
    import subprocess

    import numpy as np

    cc = shutil.which("gcc") or shutil.which("cc")
    if cc is None:
        pytest.skip("no C compiler")
    structs = [alto.alto_agg_config, alto.alto_allocator, alto.alto_batch, alto.alto_drain,
               alto._binding.alto_profile, alto.alto_split_args, alto._binding.alto_router_config,
               alto._binding.alto_routed]
    lines = ['#include <stddef.h>', '#include <stdio.h>', '#include "alto_agg.h"', 'int main(void) {']
    want = []
    for st in structs:
        name = st.__name__
        lines.append(f'  printf("%zu\\n", sizeof({name}));')
        want.append(ctypes.sizeof(st))
        for fname, _ in st._fields_:
            lines.append(f'  printf("%zu\\n", offsetof({name}, {fname}));')
            want.append(getattr(st, fname).offset)
    for dt, name in [(alto.RECORD_DTYPE, "alto_record"), (alto.PAIR_DTYPE, "alto_topk_pair")]:
        lines.append(f'  printf("%zu\\n", sizeof({name}));')
        want.append(dt.itemsize)
        for fname in dt.names:
            lines.append(f'  printf("%zu\\n", offsetof({name}, {fname}));')
            want.append(dt.fields[fname][1])
    lines += ['  return 0;', '}']
    src = tmp_path / "layout.c"
    src.write_text("\n".join(lines) + "\n")
    exe = tmp_path / "layout"
    include = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "include")
    subprocess.run([cc, "-std=c11", "-I", include, str(src), "-o", str(exe)], check=True)
    got = [int(x) for x in subprocess.run([str(exe)], check=True, capture_output=True, text=True).stdout.split()]
    assert got == want
    assert np.dtype(alto.RECORD_DTYPE).itemsize == 48


def test_constants_match_the_header():
    """Every ALTO_* constant the binding mirrors has the header's value."""
    txt = open(os.path.join(ROOT, "include", "alto_agg.h")).read()
    vals = {k: int(v, 0) for k, v in re.findall(r"#define ALTO_(\w+)\s+\(?(-?(?:0x[0-9a-fA-F]+|\d+))\)?", txt)}
    b = alto._binding
    pairs = {"ETIMEOUT": b.ETIMEOUT, "ECUDA": b.ECUDA, "MAX_DEPTH": b.MAX_DEPTH,
             "PAYLOAD_NONE": b.PAYLOAD_NONE, "PAYLOAD_CONCAT": b.PAYLOAD_CONCAT,
             "SCORE_NONE": b.SCORE_NONE, "SCORE_MAX": b.SCORE_MAX, "SCORE_TOPK": b.SCORE_TOPK,
             "FLAG_STREAM_RELEASE": b.FLAG_STREAM_RELEASE, "FLAG_DOUBLE_RING": b.FLAG_DOUBLE_RING,
             "FLAG_TEST_STALL": b.FLAG_TEST_STALL, "FLAG_DIRECT_LAUNCH": b.FLAG_DIRECT_LAUNCH,
             "OPS_PARTIAL": b.OPS_PARTIAL, "NUM_STAGES": b.NUM_STAGES, "PROFILE_OFF": b.PROFILE_OFF,
             "PROFILE_STAGES": b.PROFILE_STAGES, "PROFILE_HOT": b.PROFILE_HOT, "MAX_DELIMS": b.MAX_DELIMS,
             "ROUTE_HASH": b.ROUTE_HASH, "ROUTE_LEAST_LOADED": b.ROUTE_LEAST_LOADED}
    for name, v in pairs.items():
        assert vals[name] == v, name
    assert len(b.STAGE_NAMES) == b.NUM_STAGES
