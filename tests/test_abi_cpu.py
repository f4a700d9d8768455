"""CPU-side checks of the C ABI: the library builds for sm_103a, loads, exports every
symbol include/fk.h declares, and validates configurations on the host.  No kernel runs."""
import ctypes
import os
import re

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    from paper_2605_09681_gb300 import build, _lib
    build.build()
    return _lib.load()


def _declared():
    text = open(os.path.join(ROOT, "include", "fk.h")).read()
    return re.findall(r"FK_API\s+[\w\s\*]+?\b(fk_\w+)\s*\(", text)


def test_every_declared_symbol_is_exported(lib):
    names = _declared()
    assert len(names) >= 20
    raw = ctypes.CDLL(os.path.join(ROOT, "paper_2605_09681_gb300", "libfk.so"))
    for n in names:
        assert hasattr(raw, n), n
    from paper_2605_09681_gb300 import _lib
    assert sorted(names) == sorted(_lib.EXPORTS)


def _cfg(**kw):
    from paper_2605_09681_gb300._lib import FkConfig
    hm = np.zeros(kw.get("n_layers", 1) * kw.get("n_heads", 4), dtype=np.uint8)
    base = dict(n_layers=1, n_heads=4, head_dim=64, tokens_per_frame=60, frames_per_chunk=3,
                n_sink_frames=1, window_frames=0, n_segments=6, keep_budget_permille=700,
                select_scope=0, score_source=0, incremental=0, max_history_frames=8, device=0)
    base.update(kw)
    c = FkConfig(**base)
    c.head_is_static = hm.ctypes.data_as(ctypes.POINTER(ctypes.c_uint8))
    return c, hm


def test_config_struct_layout():
    from paper_2605_09681_gb300._lib import FkConfig
    assert ctypes.sizeof(FkConfig) == 80
    assert FkConfig.head_is_static.offset == 56
    assert (FkConfig.selection.offset, FkConfig.select_seed.offset, FkConfig.static_drop_anchor.offset,
            FkConfig.attn_precision.offset) == (64, 68, 72, 76)


def test_abi_version(lib):
    assert lib.fk_abi_version() == 4


@pytest.mark.parametrize("bad", [
    dict(head_dim=96), dict(head_dim=0), dict(n_heads=0), dict(n_heads=129), dict(n_layers=0),
    dict(n_layers=257), dict(tokens_per_frame=61), dict(n_segments=0), dict(frames_per_chunk=0),
    dict(keep_budget_permille=1001), dict(keep_budget_permille=-1), dict(select_scope=2),
    dict(score_source=5), dict(incremental=2), dict(window_frames=-1), dict(n_sink_frames=-1),
    dict(window_frames=0, max_history_frames=0), dict(selection=4), dict(selection=-1),
    dict(selection=2, select_scope=1, n_segments=1), dict(static_drop_anchor=2),
    dict(attn_precision=3), dict(attn_precision=-1), dict(attn_precision=1, head_dim=64),
    dict(attn_precision=2, head_dim=64),
])
def test_validate_rejects_bad_configs(lib, bad):
    c, _keep = _cfg(**bad)
    assert lib.fk_validate_config(ctypes.byref(c)) == 1   # FK_ERR_CONFIG


def test_validate_accepts_paper_configs(lib):
    for kw in [dict(), dict(head_dim=128, n_heads=12, tokens_per_frame=1560),
               dict(head_dim=128, n_heads=12, tokens_per_frame=8160, max_history_frames=10),
               dict(window_frames=12, keep_budget_permille=600),
               dict(n_segments=1, select_scope=1, keep_budget_permille=500, n_sink_frames=0),
               dict(n_layers=30, n_heads=12, score_source=1, incremental=1, max_history_frames=21),
               dict(selection=1, n_sink_frames=3, window_frames=4),
               dict(selection=1, window_frames=2, static_drop_anchor=1),
               dict(selection=2, n_segments=60), dict(selection=3, select_seed=7, n_segments=60),
               dict(attn_precision=1, head_dim=128), dict(attn_precision=2, head_dim=128)]:
        c, _keep = _cfg(**kw)
        assert lib.fk_validate_config(ctypes.byref(c)) == 0, kw


def test_validate_accepts_every_sweep_config(lib):
    # the seeded configurations of the GPU parity sweep, built the way the binding builds them
    from paper_2605_09681_gb300._lib import FK_ATTN, FK_SELECT, FkConfig
    import workloads as W
    from sweep_cases import N_CASES, N_LARGE, sweep_case
    cases = [sweep_case(i) for i in range(N_CASES)] + [sweep_case(i, True) for i in range(N_LARGE)]
    for w in cases:
        hm = np.ascontiguousarray(W.head_map(w).reshape(-1))
        c = FkConfig(w.n_layers, w.n_heads, w.head_dim, w.tokens_per_frame, w.frames_per_chunk,
                     w.n_sink_frames, w.window_frames, w.n_segments, w.keep_budget_permille,
                     {"per_frame": 0, "pooled": 1}[w.select_scope],
                     {"per_head": 0, "layer0_pooled": 1}[w.score_source], int(w.incremental),
                     max(1, w.max_history_frames()), 0,
                     hm.ctypes.data_as(ctypes.POINTER(ctypes.c_uint8)), FK_SELECT[w.selection],
                     w.select_seed, int(w.static_drop_anchor), FK_ATTN[w.attn_precision])
        assert lib.fk_validate_config(ctypes.byref(c)) == 0, w.name


def test_null_config_and_status_strings(lib):
    assert lib.fk_validate_config(None) == 2
    for s in range(9):
        assert lib.fk_status_str(s)
    assert lib.fk_abi_version() == 4


@pytest.mark.skipif(os.path.exists("/dev/nvidia0"), reason="checks the no-GPU error path")
def test_create_without_gpu_fails_cleanly(lib):
    c, _keep = _cfg()
    h = ctypes.c_void_p()
    st = lib.fk_create(ctypes.byref(c), ctypes.byref(h))
    assert st == 7 and not h.value          # FK_ERR_CUDA, no handle


def test_missing_library_fails_loudly(tmp_path):
    from paper_2605_09681_gb300 import _lib
    saved = _lib._lib
    _lib._lib = None
    try:
        with pytest.raises(ImportError):
            _lib.load(str(tmp_path / "libfk.so"))
    finally:
        _lib._lib = saved


def test_null_handle_calls_are_rejected(lib):
    assert lib.fk_compress(None, None) == 2
    assert lib.fk_attend(None, 0, None, None, None) == 2
    assert lib.fk_cache_bytes(None) == 0
    lib.fk_destroy(None)


def test_classify_heads_matches_oracle(lib):
    import oracle as O
    from paper_2605_09681_gb300 import classify_heads
    rng = np.random.default_rng(7)
    total = np.full(64, 100.0)
    parts = rng.dirichlet([1, 1, 1, 1], size=64) * 100.0      # gen, trans, sink, other
    mass = np.stack([total, parts[:, 0], parts[:, 1], parts[:, 2]], axis=1)
    mass[0] = [10.0, 6.0, 2.0, 0.0]                              # exactly alpha
    mass[1] = [10.0, 0.0, 0.0, 10.0]                             # all on the sinks
    for alpha in (0.5, 0.8, 0.95):
        got = classify_heads(mass, alpha)
        ref = np.array([O.classify_head(m, alpha) for m in mass], dtype=np.uint8)
        assert np.array_equal(got, ref)


def test_head_profile_rejects_bad_arguments(lib):
    # argument checks run on the host before any device query
    buf = np.zeros(4096, dtype=np.float64)
    p = buf.ctypes.data
    ok = dict(n_queries=128, n_keys=256, n_heads=2, head_dim=128, n_generate=64, n_sink=32, n_transition=32)

    def call(**kw):
        a = dict(ok, **kw)
        return lib.fk_head_profile(kw.get("Q", p), kw.get("K", p), a["n_queries"], a["n_keys"],
                                   a["n_heads"], a["head_dim"], a["n_generate"], a["n_sink"],
                                   a["n_transition"], kw.get("mass", p), kw.get("status", p), None)
    from paper_2605_09681_gb300._lib import FK_ERR_ARG, FK_ERR_CONFIG
    assert call(Q=None) == FK_ERR_ARG
    assert call(mass=None) == FK_ERR_ARG
    assert call(K=p + 8) == FK_ERR_ARG                            # not 16-byte aligned
    assert call(head_dim=96) == FK_ERR_CONFIG
    assert call(n_heads=0) == FK_ERR_CONFIG
    assert call(n_keys=0) == FK_ERR_CONFIG
    assert call(n_generate=200, n_sink=40, n_transition=40) == FK_ERR_CONFIG
    assert call(n_sink=-1) == FK_ERR_CONFIG
    assert call() == FK_ERR_ARG                                   # host pointers: not device memory


def test_quantize_e4m3_rejects_bad_arguments(lib):
    # argument checks run on the host before any device query
    buf = np.zeros(4096, dtype=np.float64)
    p = buf.ctypes.data
    e = ctypes.cast(p, ctypes.c_void_p)
    from paper_2605_09681_gb300._lib import FK_ERR_ARG, FK_ERR_CONFIG, FK_OK
    q = lib.fk_quantize_e4m3
    assert q(None, 4, 128, 1, p, e, None) == FK_ERR_ARG
    assert q(p, 4, 128, 0, None, None, None) == FK_ERR_ARG
    assert q(p + 8, 4, 128, 0, p, None, None) == FK_ERR_ARG            # not 16-byte aligned
    assert q(p, 4, 128, 1, p, None, None) == FK_ERR_ARG                # exponents required
    assert q(p, 4, 96, 1, p, e, None) == FK_ERR_CONFIG                 # scaled rows: 64 or 128
    assert q(p, 4, 12, 0, p, None, None) == FK_ERR_CONFIG              # a multiple of 8
    assert q(p, 4, 1032, 0, p, None, None) == FK_ERR_CONFIG
    assert q(p, -1, 128, 0, p, None, None) == FK_ERR_CONFIG
    assert q(p, 4, 128, 2, p, e, None) == FK_ERR_CONFIG
    assert q(p, 0, 128, 0, p, None, None) == FK_OK                     # nothing to do
    assert q(p, 4, 128, 0, p, None, None) == FK_ERR_ARG                # host pointers


def test_kernel_kinds_match_header():
    from paper_2605_09681_gb300 import KERNEL_KINDS
    text = open(os.path.join(ROOT, "include", "fk.h")).read()
    for name, v in KERNEL_KINDS.items():
        assert re.search(r"FK_KERNEL_%s = %d\b" % (name.upper(), v), text), name
    assert "FK_KERNEL_KINDS = %d" % len(KERNEL_KINDS) in text


def test_noalloc_rejects_bad_arguments_on_the_host(lib):
    # sizes beyond the documented limits and null / misaligned pointers are rejected before any
    # CUDA call (the pointer values below are never dereferenced)
    f = lib.fk_segment_scores_noalloc
    K, S = 1 << 20, 2 << 20
    assert f(None, 4, 64, 128, 8, S, None, None) == 2
    assert f(K, 4, 64, 128, 8, None, None, None) == 2
    assert f(K + 8, 4, 64, 128, 8, S, None, None) == 2            # K not 16-byte aligned
    assert f(K, 4, 64, 128, 8, S, K + 2, None) == 2               # status not 4-byte aligned
    assert f(K, 4, 64, 96, 8, S, None, None) == 1                 # head_dim
    assert f(K, 4, 64, 128, 33, S, None, None) == 1               # segments
    assert f(K, 257, 64, 128, 8, S, None, None) == 1              # frames
    assert f(K, 1, 64, 128, 8, S, None, None) == 1
    assert f(K, 256, 64, 128, 32, S, None, None) == 1             # frames x segments
    assert f(K, 4, 60, 128, 8, S, None, None) == 1                # segments must divide F


def test_stream_read_rejects_bad_arguments_on_the_host(lib):
    # null, misaligned or non-multiple-of-16 requests are refused before any CUDA call; zero
    # bytes is a no-op
    f = lib.fk_stream_read
    assert f(None, 64, None) == 2
    assert f(1 << 20 | 8, 64, None) == 2
    assert f(1 << 20, 60, None) == 2
    assert f(1 << 20, 0, None) == 0

