"""GPU parity of the CUDA path (through the C ABI) against the CPU oracle, on seeded inputs:
kept sets and scores bit-exact, attention within max abs 2e-2 / mean abs 2e-3."""
import numpy as np
import pytest

import oracle as O
import workloads as W
from fkharness import (ATOL_MAX, ATOL_MEAN, compare_layer, run_snapshot, run_stream, sample_rows,
                       snapshot, to_dev, to_f64)

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


@pytest.fixture(scope="module", autouse=True)
def _library():
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    from paper_2605_09681_gb300 import build, load_library
    build.build()
    load_library()


def _small(**kw):
    base = dict(name="small", n_layers=1, n_heads=4, head_dim=64, tokens_per_frame=60,
                frames_per_chunk=3, n_sink_frames=1, window_frames=0, n_segments=6,
                keep_budget_permille=500, schedule="snapshot", n_history_frames=7,
                static_heads=(0, 2), seed=11)
    base.update(kw)
    return W.Workload(**base)


# ------------------------------------------------------------------ small cases, every row
def test_tiny_pooled():
    run_snapshot(W.TINY)


def test_tiny_per_frame():
    run_snapshot(W.TINY_PER_FRAME)


@pytest.mark.parametrize("D", [64, 128])
@pytest.mark.parametrize("budget", [0, 333, 500, 1000])
def test_budgets_and_head_dims(D, budget):
    run_snapshot(_small(head_dim=D, keep_budget_permille=budget, seed=D + budget))


@pytest.mark.parametrize("S,nh", [(0, 1), (1, 1), (1, 2), (2, 5), (3, 3), (0, 0)])
def test_degenerate_histories(S, nh):
    # no history, sink-only history, a lone anchor, more sinks than history
    run_snapshot(_small(n_sink_frames=S, n_history_frames=nh, seed=100 + 7 * S + nh),
                 max_history_frames=max(1, nh))


def test_ragged_tiles_d128():
    # 200 tokens/frame: 600 queries (4 full q tiles + 88), segment 50, ragged key tiles
    run_snapshot(_small(head_dim=128, tokens_per_frame=200, n_segments=4, n_history_frames=9,
                        keep_budget_permille=750, seed=5))


def test_single_segment_per_frame_per_frame_scope():
    run_snapshot(_small(n_segments=1, keep_budget_permille=1000))


def test_identical_adjacent_frames_tie_break():
    # frames 1..4 identical: every score is exactly 1; ties keep the lower segment id
    w = _small(n_history_frames=6, keep_budget_permille=500)
    hk, hv, ck, cv, q = W.snapshot_inputs(w)
    F = w.tokens_per_frame
    for f in range(2, 5):
        hk[f * F:(f + 1) * F] = hk[F:2 * F]
    run_snapshot(w, inputs=(hk, hv, ck, cv, q))


def test_host_pointers_match_device():
    from paper_2605_09681_gb300 import ForcingKVCache
    w = _small(head_dim=128, tokens_per_frame=120, n_history_frames=6)
    hk, hv, ck, cv, q = W.snapshot_inputs(w)
    hm = W.head_map(w)
    outs = []
    for host in (False, True):
        with ForcingKVCache.from_workload(w, hm) as c:
            conv = (lambda a: a) if host else to_dev
            c.append_frames(0, conv(hk), conv(hv))
            c.set_current(0, conv(ck), conv(cv))
            c.compress()
            if host:
                qh = torch.from_numpy(q.view(np.int16)).view(torch.bfloat16).pin_memory()
                oh = torch.empty_like(qh).pin_memory()
                c.attend(0, qh, oh)
                torch.cuda.synchronize()
                outs.append(oh.float().numpy())
            else:
                outs.append(c.attend(0, to_dev(q)).float().cpu().numpy())
    assert np.array_equal(outs[0], outs[1])


# ------------------------------------------------------------------ streaming (window, incremental)
def test_stream_window_small():
    w = W.ROLLING.with_(name="rolling_small", head_dim=64, tokens_per_frame=48, n_heads=4,
                        window_frames=5, n_chunks=12, scene_cut_every_chunks=4)
    assert run_stream(w) == 12


@pytest.mark.parametrize("precision", ["bf16", "fp8_qk", "fp8"])
def test_heads_of_one_key_tile(precision):
    # every view fits one 128-key tile (60 current keys at the first chunk, then 100 static and
    # 120 dynamic): the attention's path with key tile 0 alone and a ragged (half-empty) tile,
    # in each precision, through appends, compressions and a sliding window
    w = W.ROLLING.with_(name="one_tile_" + precision, head_dim=128, tokens_per_frame=20, n_heads=4,
                        n_segments=4, window_frames=3, n_chunks=5, keep_budget_permille=500,
                        attn_precision=precision)
    assert run_stream(w) == 5


def test_incremental_compaction_matches_rebuild():
    # Incremental mode appends only newly decided segments into a ring of kept-segment slots;
    # the rebuild copies every kept segment each time.  The views hold the same keys in a
    # different order (the ring wraps once the 5-frame window is full): key counts agree and
    # the attention outputs agree up to summation order.
    from paper_2605_09681_gb300 import ForcingKVCache
    w = W.ROLLING.with_(name="ring", head_dim=64, tokens_per_frame=120, n_heads=4, window_frames=5,
                        n_chunks=9, scene_cut_every_chunks=4)
    hm = W.head_map(w)
    runs = []
    for inc in (True, False):
        fs = W.FrameStream(w, 0)
        res = []
        with ForcingKVCache.from_workload(w, hm, incremental=inc) as cache:
            for c in range(w.n_chunks):
                k, v = fs.frames(w.frames_per_chunk)
                cache.append_chunk(0, to_dev(k), to_dev(v))
                cache.compress()
                O = cache.attend(0, to_dev(W.queries(w, 0, c, 0)))
                res.append(([cache.key_count(0, h) for h in range(w.n_heads)],
                            [cache.kept(0, h) for h in range(w.n_heads)], to_f64(O)))
            assert cache.sync_status() == 0
        runs.append(res)
    for (ka, sa, oa), (kb, sb, ob) in zip(*runs):
        assert ka == kb and sa == sb
        err = np.abs(oa - ob)
        assert err.max() <= ATOL_MAX and err.mean() <= ATOL_MEAN / 4


def test_stream_incremental_matches_rescore():
    from paper_2605_09681_gb300 import ForcingKVCache
    w = W.ROLLING.with_(name="inc", head_dim=64, tokens_per_frame=60, n_heads=4, window_frames=6,
                        n_chunks=6)
    hm = W.head_map(w)
    got = []
    for inc in (True, False):
        fs = W.FrameStream(w, 0)
        with ForcingKVCache.from_workload(w, hm, incremental=inc) as cache:
            res = []
            for c in range(w.n_chunks):
                k, v = fs.frames(3)
                cache.append_chunk(0, to_dev(k), to_dev(v))
                cache.compress()
                res.append([(cache.kept(0, h), cache.scores(0, h)[1].tobytes()) for h in range(4)])
            got.append(res)
    assert got[0] == got[1]


@pytest.mark.parametrize("incremental", [True, False])
@pytest.mark.parametrize("D", [64, 128])
def test_stream_irregular_appends(incremental, D):
    # the current-chunk kernel forms the scoring sums of the chunk it retires when nothing else
    # touched them since the last compress; two chunk appends before one compress, or a history
    # prefill after a chunk, leave sums that match no run: they are cleared and rescored.  Kept
    # sets and scores bit-exact, attention in tolerance, at every compress.
    from paper_2605_09681_gb300 import ForcingKVCache
    w = W.ROLLING.with_(name="irregular", head_dim=D, tokens_per_frame=72, n_segments=4, n_heads=4,
                        window_frames=7, n_chunks=12, incremental=incremental, scene_cut_every_chunks=5)
    hm = W.head_map(w)
    orc = O.ForcingKVOracle.from_workload(w, hm)
    fs = W.FrameStream(w, 0)
    skip = {2, 5, 6}          # chunks appended without a compress right after them
    with ForcingKVCache.from_workload(w, hm) as cache:
        for c in range(w.n_chunks):
            if c == 8:        # a prefill of two frames after a chunk, before the compress
                k, v = fs.frames(2)
                cache.append_frames(0, to_dev(k), to_dev(v))
                orc.append_frames(0, k, v)
            k, v = fs.frames(w.frames_per_chunk)
            cache.append_chunk(0, to_dev(k), to_dev(v))
            orc.append_chunk(0, k, v)
            if c in skip:
                continue
            cache.compress()
            q = W.queries(w, 0, c, 0)
            Od = cache.attend(0, to_dev(q))
            torch.cuda.synchronize()
            compare_layer(cache, orc, 0, q, Od, label="irregular c%d" % c)
        assert cache.sync_status() == 0


def test_stream_layer0_pooled_small():
    w = W.P480_STACK.with_(name="stack_small", n_layers=3, n_heads=4, head_dim=64,
                           tokens_per_frame=60, n_chunks=5, denoise_steps=2)
    assert run_stream(w, track_layers=(0, 1, 2)) == 5 * 2 * 3


@pytest.mark.parametrize("incremental", [False, True])
def test_stream_per_head_scoring_many_layers(incremental):
    # per-head scoring in every layer, each layer with its own keys: one compress scores and
    # compacts all layers in single launches (the flattened per-layer ranges of the scoring
    # kernel, the multi-layer item list of the compaction); every layer's scores, kept sets and
    # attention are compared with its own oracle, whole-window and incremental
    w = W.P480_STACK.with_(name="layers_per_head_small", n_layers=5, n_heads=4, head_dim=128,
                           tokens_per_frame=60, n_chunks=6, denoise_steps=1,
                           score_source="per_head", incremental=incremental, window_frames=4)
    assert run_stream(w, track_layers=(0, 1, 2, 3, 4)) == 6 * 5


# ------------------------------------------------------------------ error paths (host-side)
def test_state_errors():
    from paper_2605_09681_gb300 import ForcingKVCache, FkError
    w = _small(n_history_frames=3)
    hk, hv, ck, cv, q = W.snapshot_inputs(w)
    with ForcingKVCache.from_workload(w, W.head_map(w), max_history_frames=3) as c:
        with pytest.raises(FkError) as e:
            c.attend(0, to_dev(q))
        assert e.value.name == "FK_ERR_STATE"          # no current chunk
        c.append_frames(0, to_dev(hk), to_dev(hv))
        c.set_current(0, to_dev(ck), to_dev(cv))
        with pytest.raises(FkError) as e:
            c.attend(0, to_dev(q))
        assert e.value.name == "FK_ERR_STATE"          # appended, not compressed
        c.compress()
        c.attend(0, to_dev(q))
        with pytest.raises(FkError) as e:
            c.append_chunk(0, to_dev(ck), to_dev(cv))  # history would exceed 3 frames
        assert e.value.name == "FK_ERR_FULL"
        with pytest.raises(FkError) as e:
            c.attend(7, to_dev(q))
        assert e.value.name == "FK_ERR_ARG"
        assert c.sync_status() == 0


def test_range_precondition_reported():
    from paper_2605_09681_gb300 import ForcingKVCache, STATUS_NAMES
    w = _small(n_history_frames=4)
    hk, hv, ck, cv, q = W.snapshot_inputs(w)
    big = W.to_bf16_bits(np.full(hk.shape, 400.0))      # n_p = 64 * 400^2 > 2^23
    with ForcingKVCache.from_workload(w, W.head_map(w)) as c:
        c.append_frames(0, to_dev(big), to_dev(hv))
        c.set_current(0, to_dev(ck), to_dev(cv))
        c.compress()
        assert STATUS_NAMES[c.sync_status()] == "FK_ERR_RANGE"
        assert c.sync_status() == 0                     # the status word is cleared


# ------------------------------------------------------------------ full-size workloads
def test_480p_layer():
    # every query row of every head: all 19 query-tile pairs of each of the 12 heads
    st = run_snapshot(W.P480_LAYER)
    print("480p", st)


def test_1080p_layer():
    # sampled rows of every head, then every row of the first static and the first dynamic head
    # (all 96 query-tile pairs of each)
    w = W.P1080_LAYER
    hm = W.head_map(w)[0]
    full = [int(np.flatnonzero(hm == 1)[0]), int(np.flatnonzero(hm == 0)[0])]
    st = run_snapshot(w, rows=sample_rows(w.n_queries, 64), full_heads=full)
    print("1080p", st)


def test_contract_golden_tokens_on_gpu():
    # the hand-worked tokens of tests/golden/contract_token_dot.txt through the GPU scorer: one
    # token per segment, frame 0 = the a rows, frame 1 = the b rows, frame 2 = zeros.  Every
    # self-dot is 2^21, so s_0^(j) = d_j 2^24 / (2^21 2^24) = d_j 2^-21 (the hand value), and
    # frame 1 against the zero frame scores 0.
    from paper_2605_09681_gb300 import ForcingKVCache
    from test_oracle_pins import _contract_golden
    toks = _contract_golden()
    for D in (64, 128):
        rows = [t for t in toks if t[1] == D]
        n = len(rows)
        frames = np.zeros((3, n, 1, D), dtype=np.float32)
        for j, (_name, _D, a, b, _v) in enumerate(rows):
            frames[0, j, 0], frames[1, j, 0] = a, b
        kb = W.to_bf16_bits(frames.reshape(3 * n, 1, D))
        kd = to_dev(kb)
        with ForcingKVCache(n_layers=1, n_heads=1, head_dim=D, tokens_per_frame=n, frames_per_chunk=1,
                            n_sink_frames=0, window_frames=0, n_segments=n, keep_budget_permille=500,
                            head_is_static=[[0]], max_history_frames=3) as c:
            c.append_frames(0, kd, kd)
            c.compress()
            first, sc = c.scores(0, 0)
            assert c.sync_status() == 0
        assert first == 0 and sc.shape == (2, n)
        want = np.array([[v["contract"] * 2.0 ** -21 for *_x, v in rows], [0.0] * n], dtype=np.float32)
        assert np.array_equal(sc.view(np.uint32), want.view(np.uint32)), (D, sc, want)


def test_rolling_full():
    w = W.ROLLING
    assert run_stream(w, compare_every=10) >= 6


def test_480p_stack_full():
    # all 30 layers are appended and compressed; layers 0, 13, 29 carry their own seeded
    # data and are attended and compared (the other layers replay layer 0's inputs)
    w = W.P480_STACK
    assert run_stream(w, track_layers=(0, 13, 29), compare_every=3, step_filter=(0, 3)) > 0


def _check_head_profile(q, k, g, s, t):
    """Eq. 1 masses of the GPU kernel vs the fp64 oracle on the same bf16 inputs; the
    classification of every head not within 1e-3 of the threshold; a second call adds to the
    same accumulator."""
    from paper_2605_09681_gb300 import classify_heads, head_profile
    H = q.shape[1]
    Qd, Kd = to_dev(q), to_dev(k)
    mass, status = head_profile(Qd, Kd, g, s, t)
    torch.cuda.synchronize()
    got = mass.cpu().numpy()
    assert int(status.item()) == 0
    Qf, Kf = W.bf16_bits_to_f32(q), W.bf16_bits_to_f32(k)
    ref = np.stack([O.head_attention_mass(Qf[:, h], Kf[:, h], g, s, t) for h in range(H)])
    nq = q.shape[0]
    assert np.all(got[:, 0] == nq)
    assert np.abs(got - ref).max() <= 1e-4 * nq, np.abs(got - ref).max()
    ratio = (ref[:, 1] + ref[:, 2]) / (ref[:, 0] - ref[:, 3])
    clear = np.abs(ratio - 0.8) > 1e-3
    assert np.array_equal(classify_heads(got, 0.8)[clear],
                          np.array([O.classify_head(m, 0.8) for m in ref], dtype=np.uint8)[clear])
    head_profile(Qd, Kd, g, s, t, mass=mass, status=status)
    torch.cuda.synchronize()
    assert np.allclose(mass.cpu().numpy(), 2 * got, rtol=1e-12, atol=0)


@pytest.mark.parametrize("head_dim,F,hist", [(128, 260, 8), (64, 100, 5), (128, 24, 2), (64, 40, 2)])
def test_head_profile_matches_oracle(head_dim, F, hist):
    # 3-frame chunk, ragged query and key tiles, class boundaries inside key tiles.  The two
    # CTAs of a cluster split the key tiles: 27 (13 + 14), 8, a single tile (the first CTA has
    # none) and two tiles (one each, the second ragged).
    q, k, (g, s, t) = W.profile_inputs(11 + head_dim, 8, head_dim, F, 3, 1, hist)
    _check_head_profile(q, k, g, s, t)


@pytest.mark.parametrize("i", range(16))
def test_head_profile_sweep(i):
    # seeded draws of heads (1-12), head_dim, tokens per frame (8-300), chunk frames (1-3),
    # sink frames (0-2, so an empty sink class too) and other history frames (0-7): query
    # tiles, key tiles, the cluster's key split and the class boundaries land anywhere
    rng = np.random.default_rng(3571 * (i + 1))
    H, D = int(rng.integers(1, 13)), int(rng.choice([64, 128]))
    F, C, S = int(rng.integers(8, 301)), int(rng.integers(1, 4)), int(rng.integers(0, 3))
    hist = S + 1 + int(rng.integers(0, 8))
    q, k, (g, s, t) = W.profile_inputs(200 + i, H, D, F, C, S, hist)
    _check_head_profile(q, k, g, s, t)


def test_host_inputs_and_overlap_match_device_inputs():
    # the same stream driven with device tensors; with pageable host arrays (inputs copied
    # in call order, output copied back); and with pinned host tensors and host-input overlap
    # on (inputs copied on the handle's copy stream into two alternating staging slots).  The
    # overlap run issues every step
    # before one final synchronize, so copies into a slot really race the kernels still
    # reading the other slot.  All three produce bit-identical outputs.
    from paper_2605_09681_gb300 import ForcingKVCache
    w = W.ROLLING.with_(name="ovl", head_dim=64, tokens_per_frame=120, n_heads=4, window_frames=6,
                        n_chunks=7)
    hm = W.head_map(w)
    pin = lambda a: torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).view(torch.bfloat16).pin_memory()
    runs = {}
    for mode in ("device", "host", "overlap"):
        fs = W.FrameStream(w, 0)
        keep, outs = [], []
        with ForcingKVCache.from_workload(w, hm) as cache:
            cache.set_host_overlap(mode == "overlap")
            for c in range(w.n_chunks):
                k, v = fs.frames(w.frames_per_chunk)
                q = W.queries(w, 0, c, 0)
                if mode == "device":
                    cache.append_chunk(0, to_dev(k), to_dev(v))
                    cache.compress()
                    outs.append(cache.attend(0, to_dev(q)))
                else:
                    if mode == "host":
                        K, V, Q = (np.ascontiguousarray(x) for x in (k, v, q))
                        Oh = np.zeros(q.shape, dtype=np.uint16)
                    else:
                        K, V, Q = pin(k), pin(v), pin(q)
                        Oh = torch.empty(Q.shape, dtype=torch.bfloat16).pin_memory()
                    keep += [K, V, Q]
                    cache.append_chunk(0, K, V)
                    cache.compress()
                    cache.set_current(0, K, V)
                    cache.attend(0, Q, Oh)
                    outs.append(Oh)
                    if mode == "host":
                        torch.cuda.synchronize()
            cache.wait_outputs()
            torch.cuda.current_stream().synchronize()   # stream order alone covers the outputs
            assert cache.sync_status() == 0
            runs[mode] = [W.bf16_bits_to_f32(o) if isinstance(o, np.ndarray) else o.float().cpu().numpy()
                          for o in outs]
    for a, b, c in zip(runs["device"], runs["host"], runs["overlap"]):
        assert np.array_equal(a, b) and np.array_equal(a, c)


@pytest.mark.parametrize("name", ["full_kv_480p", "streamingllm_480p", "dummy_forcing_480p",
                                  "uniform_tokens_480p", "random_tokens_480p"])
def test_comparison_rules_480p(name):
    # the paper's comparison rules through the same selection, compaction and attention
    # kernels: kept sets and ranking values bit-exact, attention within tolerance
    w = W.WORKLOADS[name]
    run_snapshot(w, rows=sample_rows(w.n_queries, 64))


def test_bounded_wait_expiry_is_reported_and_context_survives():
    # a wait on an mbarrier that nothing completes gives up after its limit, the status word
    # reports FK_ERR_TIMEOUT once, and the same handle then runs the hot path normally
    from paper_2605_09681_gb300 import ForcingKVCache
    from paper_2605_09681_gb300._lib import FK_ERR_TIMEOUT
    import time
    w = W.TINY_PER_FRAME
    hm = W.head_map(w)
    with ForcingKVCache.from_workload(w, hm) as cache:
        t0 = time.perf_counter()
        cache.wait_selftest(20000)                   # 20 ms
        assert cache.sync_status() == FK_ERR_TIMEOUT
        assert time.perf_counter() - t0 >= 0.019
        assert cache.sync_status() == 0              # cleared once read
    run_snapshot(w)                                  # the context is still usable
