"""Pins of the CPU oracle to facts fixed outside it: hand-worked index sets from Eq. 2,
closed forms, an independent fmaf (the C library's), library routines (scipy cosine,
torch scaled_dot_product_attention), exact integer arithmetic, brute-force enumeration
and invariants.  CPU only."""
import ctypes
import ctypes.util
import itertools
import math
import os

import numpy as np
import pytest
import torch

import oracle as O
import workloads as W

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _rng(seed=0):
    return np.random.default_rng(seed)


def _bf16(x):
    return W.bf16_bits_to_f32(W.to_bf16_bits(np.asarray(x, dtype=np.float64)))


def _parse_range(s):
    s = s.strip()
    if s == "-":
        return ()
    out = []
    for part in s.split(","):
        if "-" in part:
            a, b = part.split("-")
            out += list(range(int(a), int(b) + 1))
        else:
            out.append(int(part))
    return tuple(out)


# ---------------------------------------------------------------- frame bookkeeping
def test_frame_roles_golden():
    n = 0
    for line in open(os.path.join(GOLDEN, "frame_roles.txt")):
        if line.startswith("#") or not line.strip():
            continue
        cols = [c.strip() for c in line.split("|")]
        nh, S, Wn = map(int, cols[0].split())
        r = O.frame_roles(nh, S, Wn)
        assert r.sink == _parse_range(cols[1]), line
        assert r.window == _parse_range(cols[2]), line
        anchor = None if cols[3] == "-" else int(cols[3])
        assert r.anchor == anchor, line
        assert r.scoreable == _parse_range(cols[4]), line
        n += 1
    assert n >= 8


def test_eq2_static_tokens_golden():
    lines = [l for l in open(os.path.join(GOLDEN, "eq2_static_tokens.txt")) if not l.startswith("#")]
    params = dict(kv.split("=") for kv in lines[0].split())
    C, F, S, i = (int(params[k]) for k in ("C", "F", "S", "i"))
    expected = [int(x) for x in lines[1].split()]
    roles = O.frame_roles(i * C, S, 0)
    got = O.static_key_tokens(roles, F, range(i * C, (i + 1) * C))
    assert got == expected


def test_segment_ranges_partition_frame():
    for F, n in [(60, 1), (60, 6), (1560, 6), (8160, 6), (12, 4)]:
        rs = [O.segment_range(F, n, j) for j in range(n)]
        assert rs[0][0] == 0 and rs[-1][1] == F
        assert all(a[1] == b[0] for a, b in zip(rs, rs[1:]))
        assert len({hi - lo for lo, hi in rs}) == 1
    with pytest.raises(ValueError):
        O.segment_range(10, 3, 0)


def test_keep_count_floor():
    assert O.keep_count(700, 6) == 4      # b = 1 - r = 0.7 with r = 0.3, n = 6 (App. H)
    assert O.keep_count(600, 6) == 3
    assert O.keep_count(500, 6) == 3
    assert O.keep_count(500, 1) == 0
    assert O.keep_count(1000, 6) == 6
    assert O.keep_count(0, 6) == 0
    assert O.keep_count(300, 6) == 1      # Eq. 3 literally: floor(r n) with r = 0.3


# ---------------------------------------------------------------- Eq. 3 scores
def test_fmaf_emulation_matches_c_library():
    libm = ctypes.CDLL(ctypes.util.find_library("m"))
    libm.fmaf.restype = ctypes.c_float
    libm.fmaf.argtypes = [ctypes.c_float] * 3
    rng = _rng(1)
    a = _bf16(rng.standard_normal(4000) * np.exp2(rng.integers(-20, 20, 4000)))
    b = _bf16(rng.standard_normal(4000) * np.exp2(rng.integers(-20, 20, 4000)))
    c = (rng.standard_normal(4000) * np.exp2(rng.integers(-40, 40, 4000))).astype(np.float32)
    got = O.fmaf_bf16(a, b, c)
    ref = np.array([libm.fmaf(float(x), float(y), float(z)) for x, y, z in zip(a, b, c)],
                   dtype=np.float32)
    assert np.array_equal(got.view(np.uint32), ref.view(np.uint32))


@pytest.mark.parametrize("D", [64, 128])
def test_token_dot_exact_on_small_integers(D):
    rng = _rng(D)
    A = rng.integers(-8, 9, size=(300, D)).astype(np.float32)
    B = rng.integers(-8, 9, size=(300, D)).astype(np.float32)
    exact = (A.astype(np.int64) * B.astype(np.int64)).sum(axis=1)
    assert np.array_equal(O.token_dots_contract(A, B).astype(np.int64), exact)


@pytest.mark.parametrize("D", [64, 128])
def test_token_dot_within_fp32_error_bound(D):
    # an fma chain of 8 then log2(D/8) butterfly adds: error <= (8 + log2(D/8)) u sum|ab|
    rng = _rng(D + 1)
    A = _bf16(rng.standard_normal((2000, D)) * 3)
    B = _bf16(rng.standard_normal((2000, D)) * 3)
    exact = (A.astype(np.float64) * B.astype(np.float64)).sum(axis=1)
    bound = (8 + math.log2(D // 8)) * 2.0 ** -24 * np.abs(A.astype(np.float64) * B).sum(axis=1)
    err = np.abs(O.token_dots_contract(A, B).astype(np.float64) - exact)
    assert (err <= bound * 1.0001 + 1e-30).all()


def _contract_golden():
    """Tokens of tests/golden/contract_token_dot.txt: (name, D, a, b, values by column)."""
    cols = ("contract", "exact", "rev", "strd", "desc", "last2", "first2", "short", "n_a", "n_b")
    out = []
    for line in open(os.path.join(GOLDEN, "contract_token_dot.txt")):
        line = line.split("#")[0].strip()
        if not line:
            continue
        head, a_s, b_s, vals, alts, norms = (p.strip() for p in line.split("|"))
        name, D = head.split()
        D = int(D)
        vec = []
        for spec in (a_s, b_s):
            v = np.zeros(D, dtype=np.float32)
            for item in spec.split():
                c, x = item.split(":")
                v[int(c)] = float(x)
            vec.append(v)
        nums = [float(x) for x in (vals + " " + alts + " " + norms).split()]
        out.append((name, D, vec[0], vec[1], dict(zip(cols, nums))))
    return out


def _dot_in_order(a, b, D, variant):
    """The per-token dot under the contract ("contract") or one of the misreadings recorded in
    the golden file, for inputs whose products are exact (fp64 sums of them are exact too)."""
    G = D // 8
    groups = [list(range(8 * g, 8 * g + 8)) for g in range(G)]
    if variant == "strd":
        groups = [[g + G * i for i in range(8)] for g in range(G)]
    if variant == "desc":
        groups = [grp[::-1] for grp in groups]
    p = []
    for grp in groups:
        acc = np.float32(0.0)
        for c in grp:
            acc = np.float32(float(a[c]) * float(b[c]) + float(acc))
        p.append(acc)
    strides = [G >> k for k in range(1, G.bit_length())]      # G/2, ..., 2, 1
    if variant == "rev":
        strides = strides[::-1]
    elif variant == "last2":
        strides = strides[:-2] + [strides[-1], strides[-2]]
    elif variant == "first2":
        strides = [strides[1], strides[0]] + strides[2:]
    elif variant == "short":
        strides = strides[1:]
    for s in strides:
        p = [np.float32(p[g] + p[g ^ s]) for g in range(G)]
    return float(p[0])


def test_contract_token_dot_golden():
    # hand-worked values (tests/golden/contract_token_dot.txt): the oracle's per-token dot and
    # self-dots equal them bit for bit, so a reordered butterfly or a regrouped / reversed fma
    # chain in the oracle fails here
    toks = _contract_golden()
    assert {D for _, D, *_ in toks} == {64, 128}
    for name, D, a, b, v in toks:
        A, B = a[None, :], b[None, :]
        assert O.token_dots_contract(A, B)[0] == np.float32(v["contract"]), name
        assert O.token_dots_contract(A, A)[0] == np.float32(v["n_a"]), name
        assert O.token_dots_contract(B, B)[0] == np.float32(v["n_b"]), name
        assert float(np.dot(a.astype(np.float64), b.astype(np.float64))) == v["exact"], name
        # a one-token segment pair: N1 = n_a 2^24, N2 = n_b 2^24, Dsum = d 2^24, so
        # s = d / sqrt(n_a n_b) exactly (here d 2^-21: 2^-24 or 2^-25)
        s = O.segment_score_contract(A, B)
        assert s == np.float32(v["contract"] / math.sqrt(v["n_a"] * v["n_b"])), name


def test_contract_golden_file_is_consistent_and_discriminating():
    # the recorded misreadings are what those orders give (each row's hand derivation is
    # replayed in plain fp32 steps), and every misreading changes at least one token per D
    toks = _contract_golden()
    variants = ("rev", "strd", "desc", "last2", "first2", "short")
    for name, D, a, b, v in toks:
        assert _dot_in_order(a, b, D, "contract") == v["contract"], name
        for var in variants:
            assert _dot_in_order(a, b, D, var) == v[var], (name, var)
    for D in (64, 128):
        rows = [v for _, d, _, _, v in toks if d == D]
        for var in variants:
            assert any(r[var] != r["contract"] for r in rows), (D, var)


def test_fixed_point_truncates_toward_zero():
    x = np.array([1.5, -1.5, 2.0 ** -25, -(2.0 ** -25), 3.0, 0.0], dtype=np.float64) * 2.0 ** -24
    assert O.fixed_point(x).tolist() == [1, -1, 0, 0, 3, 0]
    assert O.fixed_point(np.float32(2.0 ** 23)).item() == 2 ** 47


def test_score_closed_forms():
    rng = _rng(3)
    a = _bf16(rng.standard_normal((260, 128)))
    assert O.segment_score_contract(a, a) == np.float32(1.0)
    assert O.segment_score_contract(a, -a) == np.float32(-1.0)
    # disjoint channel support in every token: orthogonal segments
    b = a.copy()
    a2 = a.copy()
    a2[:, 64:] = 0
    b[:, :64] = 0
    assert O.segment_score_contract(a2, b) == np.float32(0.0)
    assert O.segment_score_contract(np.zeros_like(a), a) == np.float32(0.0)
    assert O.cosine_fp64(a2, b) == 0.0
    assert abs(O.cosine_fp64(a, -a) + 1.0) < 1e-15


def test_cosine_matches_scipy_and_contract():
    from scipy.spatial.distance import cosine as scipy_cosine
    rng = _rng(4)
    for rho in (0.0, 0.5, 0.9, 0.99):
        x = _bf16(rng.standard_normal((260, 128)) * 1.7)
        y = _bf16(rho * x + math.sqrt(1 - rho * rho) * rng.standard_normal((260, 128)) * 1.7)
        ref = 1.0 - scipy_cosine(x.astype(np.float64).ravel(), y.astype(np.float64).ravel())
        assert abs(O.cosine_fp64(x, y) - ref) < 1e-12
        assert abs(float(O.segment_score_contract(x, y)) - ref) <= 1e-6


def test_contract_scores_token_permutation_invariant():
    rng = _rng(5)
    x = _bf16(rng.standard_normal((260, 128)))
    y = _bf16(0.9 * x + 0.4 * rng.standard_normal((260, 128)))
    p = rng.permutation(260)
    s0 = O.segment_score_contract(x, y)
    s1 = O.segment_score_contract(x[p], y[p])
    assert s0.view(np.uint32) == s1.view(np.uint32)


def test_cosine_scale_invariant_fp64():
    rng = _rng(6)
    x = _bf16(rng.standard_normal((100, 64)))
    y = _bf16(rng.standard_normal((100, 64)) + x)
    for m in (-3, 2, 5):
        assert abs(O.cosine_fp64(x * 2.0 ** m, y) - O.cosine_fp64(x, y)) < 1e-14


def test_score_precondition_enforced():
    a = np.full((4, 128), 300.0, dtype=np.float32)   # n_p = 128 * 90000 > 2^23
    with pytest.raises(ValueError):
        O.segment_score_contract(a, a)


# ---------------------------------------------------------------- Eq. 3 BottomK
def _brute_force_keep(scores, k):
    """The unique size-k subset whose members all precede every non-member in (score, index)."""
    n = len(scores)
    key = [(float(s), i) for i, s in enumerate(scores)]
    hits = []
    for sub in itertools.combinations(range(n), k):
        rest = [i for i in range(n) if i not in sub]
        if all(key[a] < key[b] for a in sub for b in rest):
            hits.append(sorted(sub))
    assert len(hits) == 1
    return hits[0]


def test_bottom_k_brute_force_with_ties():
    rng = _rng(7)
    for trial in range(300):
        n = int(rng.integers(1, 8))
        s = rng.choice(np.array([0.1, 0.5, 0.5, 0.9, -0.2, 0.5], dtype=np.float32), size=n)
        for k in range(n + 1):
            assert O.bottom_k(s, range(n), k) == _brute_force_keep(s, k)


def test_bottom_k_keeps_lowest_similarity():
    s = np.array([0.99, 0.2, 0.95, 0.1, 0.97, 0.5], dtype=np.float32)
    # evict the highest-similarity segments, keep floor(0.7 * 6) = 4 (Sec. 4.3)
    assert O.bottom_k(s, range(6), 4) == [1, 2, 3, 5]


def test_bottom_k_ties_go_to_lower_index():
    s = np.float32([0.5] * 6)
    assert O.bottom_k(s, range(6), 3) == [0, 1, 2]


# ---------------------------------------------------------------- Eq. 3/4 on constructed frames
def _constructed_oracle(static_map, n_hist=5, S=1, C=2, F=12, n=4, D=64, budget=500, seed=8):
    """Frames whose segments j in `same[t]` are copied from frame t into frame t+1."""
    rng = _rng(seed)
    H = len(static_map)
    frames = [rng.standard_normal((F, H, D))]
    same = {}
    for t in range(1, n_hist + C):
        f = rng.standard_normal((F, H, D))
        pick = rng.choice(n, size=n - O.keep_count(budget, n), replace=False)
        same[t - 1] = sorted(pick.tolist())
        for j in pick:
            lo, hi = O.segment_range(F, n, j)
            f[lo:hi] = frames[-1][lo:hi]
        frames.append(f)
    bits = W.to_bf16_bits(np.concatenate(frames))
    orc = O.ForcingKVOracle(n_layers=1, n_heads=H, head_dim=D, tokens_per_frame=F,
                            frames_per_chunk=C, n_sink_frames=S, window_frames=0, n_segments=n,
                            keep_budget_permille=budget, head_is_static=[static_map])
    orc.append_frames(0, bits[:n_hist * F], bits[:n_hist * F])
    orc.append_chunk(0, bits[n_hist * F:], bits[n_hist * F:])
    return orc, same


def test_kept_segments_are_the_changed_ones():
    orc, same = _constructed_oracle([0, 0])
    n = 4
    for h in range(2):
        sc = orc.scores(0, h)
        kept = orc.kept(0, h)
        for t in orc.roles(0).scoreable:
            for j in same[t]:
                assert sc[t][j] == np.float32(1.0)       # t compared with t+1, not t-1
            expect = [t * n + j for j in range(n) if j not in same[t]]
            assert [s for s in kept if s // n == t] == expect


def test_dynamic_set_full_budget_is_full_window():
    orc, _ = _constructed_oracle([0, 1], budget=1000)
    total = (orc.nh[0] + orc.C) * orc.F
    assert sorted(orc.key_tokens(0, 0)) == list(range(total))


def test_dynamic_set_zero_budget_is_static_set():
    orc, _ = _constructed_oracle([0, 1], budget=0)
    assert orc.key_tokens(0, 0) == orc.key_tokens(0, 1)
    roles = orc.roles(0)
    assert orc.key_tokens(0, 1) == O.static_key_tokens(roles, orc.F, orc.current_frames(0))


def test_pooled_selection_brute_force():
    w = W.TINY
    hk, hv, ck, cv, q = W.snapshot_inputs(w)
    orc = O.ForcingKVOracle.from_workload(w, W.head_map(w))
    orc.append_frames(0, hk, hv)
    orc.append_chunk(0, ck, cv)
    for h in (2, 3):
        sc = orc.scores(0, h)
        flat = np.array([sc[t][0] for t in sorted(sc)])
        assert len(flat) == 6
        assert orc.kept(0, h) == _brute_force_keep(flat, 3)


def test_layer0_pooled_score_is_cosine_over_heads():
    w = W.TINY_PER_FRAME.with_(score_source="layer0_pooled", n_layers=2)
    fs = W.FrameStream(w, 0)
    hk, hv = fs.frames(w.n_history_frames)
    orc = O.ForcingKVOracle.from_workload(w, W.head_map(w))
    orc.append_frames(0, hk, hv)
    sc = orc.scores(1, 2)  # a layer-1 dynamic head is scored with layer-0 keys of all heads
    K = W.bf16_bits_to_f32(hk).reshape(w.n_history_frames, w.tokens_per_frame, w.n_heads, w.head_dim)
    for t in sc:
        for j in range(w.n_segments):
            lo, hi = O.segment_range(w.tokens_per_frame, w.n_segments, j)
            ref = O.cosine_fp64(K[t, lo:hi], K[t + 1, lo:hi])
            assert abs(float(sc[t][j]) - ref) <= 1e-6


# ---------------------------------------------------------------- attention
def _sdpa64(Q, K, V):
    q = torch.from_numpy(np.asarray(Q, np.float64))[None, None]
    k = torch.from_numpy(np.asarray(K, np.float64))[None, None]
    v = torch.from_numpy(np.asarray(V, np.float64))[None, None]
    return torch.nn.functional.scaled_dot_product_attention(q, k, v)[0, 0].numpy()


def test_attention_matches_torch_sdpa():
    rng = _rng(9)
    Q, K, V = (rng.standard_normal((300, 64)), rng.standard_normal((777, 64)) * 2,
               rng.standard_normal((777, 64)))
    assert np.abs(O.attention_fp64(Q, K, V, row_block=64) - _sdpa64(Q, K, V)).max() < 1e-12


def test_attention_closed_forms():
    rng = _rng(10)
    Q = rng.standard_normal((5, 32))
    K1, V1 = rng.standard_normal((1, 32)), rng.standard_normal((1, 32))
    assert np.allclose(O.attention_fp64(Q, K1, V1), np.repeat(V1, 5, 0), atol=1e-15)
    Ks = np.repeat(rng.standard_normal((1, 32)), 40, 0)
    V = rng.standard_normal((40, 32))
    assert np.allclose(O.attention_fp64(Q, Ks, V), V.mean(0, keepdims=True), atol=1e-13)


def test_oracle_full_budget_equals_full_attention():
    w = W.TINY_PER_FRAME.with_(keep_budget_permille=1000)
    hk, hv, ck, cv, q = W.snapshot_inputs(w)
    orc = O.ForcingKVOracle.from_workload(w, W.head_map(w))
    orc.append_frames(0, hk, hv)
    orc.append_chunk(0, ck, cv)
    out = orc.attend(0, q)
    Kall = W.bf16_bits_to_f32(np.concatenate([hk, ck]))
    Vall = W.bf16_bits_to_f32(np.concatenate([hv, cv]))
    Qf = W.bf16_bits_to_f32(q)
    for h in (2, 3):   # dynamic heads: full window
        ref = _sdpa64(Qf[:, h], Kall[:, h], Vall[:, h])
        assert np.abs(out[:, h] - ref).max() < 1e-12
    F = w.tokens_per_frame
    for h in (0, 1):   # static heads: Eq. 2 only (no sink in this case: anchor + chunk)
        idx = np.r_[6 * F:7 * F, 7 * F:10 * F]
        ref = _sdpa64(Qf[:, h], Kall[idx, h], Vall[idx, h])
        assert np.abs(out[:, h] - ref).max() < 1e-12


def test_view_lengths_match_paper_sizes():
    # 480P single layer: static = sink + anchor + chunk, dynamic adds 17 frames x 4 x 260 tokens
    w = W.P480_LAYER
    roles = O.frame_roles(w.n_history_frames, w.n_sink_frames, w.window_frames)
    F = w.tokens_per_frame
    cur = range(19, 22)
    assert len(O.static_key_tokens(roles, F, cur)) == 7800
    kept = [t * 6 + j for t in roles.scoreable for j in range(4)]
    assert len(O.dynamic_key_tokens(roles, F, 6, kept, cur)) == 25480


def test_window_drops_old_frames():
    w = W.ROLLING.with_(tokens_per_frame=12, n_heads=2, head_dim=16, n_chunks=8)
    orc = O.ForcingKVOracle.from_workload(w, [[1, 0]])
    fs = W.FrameStream(w, 0)
    for c in range(8):
        k, v = fs.frames(3)
        orc.append_chunk(0, k, v)
    r = orc.roles(0)
    assert orc.nh[0] == 21 and r.window == tuple(range(9, 21)) and r.sink == (0,)
    assert sorted(orc.frames[0]) == [0] + list(range(9, 21))
    assert len(orc.kept(0, 1)) == 11 * 3


# ---- offline head profiling (Sec. 4.1, Eq. 1)

def _class_layout(n_gen, n_sink, n_other, n_trans, D, seed):
    rng = np.random.default_rng(seed)
    return rng.standard_normal((n_gen + n_sink + n_other + n_trans, D))


def test_head_mass_uniform_attention_closed_form():
    # q = 0: every logit is 0, each row spreads its unit mass evenly over the Nk keys, so each
    # class receives rows * (class size) / Nk exactly
    n_gen, n_sink, n_other, n_trans, D, nq = 30, 10, 45, 15, 16, 7
    K = _class_layout(n_gen, n_sink, n_other, n_trans, D, 0)
    nk = K.shape[0]
    m = O.head_attention_mass(np.zeros((nq, D)), K, n_gen, n_sink, n_trans)
    assert np.allclose(m, [nq, nq * n_gen / nk, nq * n_trans / nk, nq * n_sink / nk], rtol=0, atol=1e-12)


def test_head_mass_two_key_values_closed_form():
    # keys take two values: a on the generated chunk, b everywhere else; one query row q.
    # The softmax is then n_gen e^{q.a/s} / Z on the chunk and e^{q.b/s} / Z on each other key.
    D = 8
    n_gen, n_sink, n_other, n_trans = 5, 3, 7, 4
    a = np.linspace(-1, 1, D)
    b = np.cos(np.arange(D))
    q = np.sin(np.arange(D) * 0.7)
    K = np.vstack([np.tile(a, (n_gen, 1)), np.tile(b, (n_sink + n_other + n_trans, 1))])
    ea, eb = np.exp(q @ a / np.sqrt(D)), np.exp(q @ b / np.sqrt(D))
    Z = n_gen * ea + (n_sink + n_other + n_trans) * eb
    m = O.head_attention_mass(q[None], K, n_gen, n_sink, n_trans)
    assert np.allclose(m, [1.0, n_gen * ea / Z, n_trans * eb / Z, n_sink * eb / Z], rtol=1e-13, atol=0)


def test_head_mass_class_boundaries_and_permutations():
    # shuffling keys inside a class leaves the masses unchanged; moving one key across a
    # class boundary changes exactly the two classes involved
    n_gen, n_sink, n_other, n_trans, D = 12, 6, 20, 6, 16
    rng = np.random.default_rng(3)
    K = _class_layout(n_gen, n_sink, n_other, n_trans, D, 1)
    Q = rng.standard_normal((9, D)) * 2.0
    m = O.head_attention_mass(Q, K, n_gen, n_sink, n_trans)
    P = K.copy()
    P[:n_gen] = P[rng.permutation(n_gen)]
    P[n_gen + n_sink + n_other:] = P[n_gen + n_sink + n_other + rng.permutation(n_trans)]
    assert np.allclose(O.head_attention_mass(Q, P, n_gen, n_sink, n_trans), m, rtol=1e-13, atol=1e-13)
    m2 = O.head_attention_mass(Q, K, n_gen + 1, n_sink - 1, n_trans)   # key n_gen: sink -> generated
    logits = Q @ K.T / np.sqrt(D)
    p = np.exp(logits - logits.max(1, keepdims=True))
    p /= p.sum(1, keepdims=True)
    moved = p[:, n_gen].sum()
    assert np.isclose(m2[1] - m[1], moved, rtol=1e-12) and np.isclose(m[3] - m2[3], moved, rtol=1e-12)
    assert m2[0] == m[0] and m2[2] == m[2]


def test_classify_head_threshold():
    # Eq. 1 with alpha = 0.8: (gen + trans) / (total - sink)
    assert O.classify_head([10.0, 6.0, 2.0, 1.0], 0.8)          # 8/9 = 0.889 > 0.8: static
    assert not O.classify_head([10.0, 4.0, 2.0, 1.0], 0.8)      # 6/9 = 0.667: dynamic
    assert not O.classify_head([10.0, 6.0, 2.0, 0.0], 0.8)      # exactly 0.8 is not above it
    assert O.classify_head([10.0, 0.0, 0.0, 10.0], 0.8)         # all mass on the sinks


# ---- comparison selection rules (App. H, Sec. 5.3)

def test_splitmix64_published_vector():
    # first output of SplitMix64 from state 0 (the generator's published reference output)
    assert O.splitmix64(0) == 0xE220A8397B1DCDAF


def test_rule_uniform_keeps_evenly_spaced_segments():
    for n, k in [(6, 4), (6, 3), (1560, 1092), (10, 10), (7, 1)]:
        kept = [j for j in range(n) if O.rule_value("uniform", 0, 3, j, n, k) == 0.0]
        assert kept == sorted({i * n // k for i in range(k)}) and len(kept) == k
    assert O.rule_value("uniform", 0, 0, 0, 6, 0) == 1.0


def test_rule_random_is_seeded_uniform():
    vals = np.array([O.rule_value("random", 7, t, j, 1560, 1092) for t in range(3) for j in range(1560)])
    assert np.all((vals >= 0) & (vals < 1)) and abs(vals.mean() - 0.5) < 0.02
    assert np.all(vals * 16777216 == np.floor(vals * 16777216))          # 24-bit values
    again = [O.rule_value("random", 7, 1, j, 1560, 1092) for j in range(5)]
    other = [O.rule_value("random", 8, 1, j, 1560, 1092) for j in range(5)]
    assert again == [O.rule_value("random", 7, 1, j, 1560, 1092) for j in range(5)] and again != other


def test_rule_workloads_key_sets():
    # StreamingLLM: every head = 3 sinks + 4 recent frames + chunk; Dummy Forcing L = 2:
    # local heads = sink + chunk, neighbour heads = sink + 2 recent frames + chunk
    F = 12
    for w, want_static, want_dynamic in [
            (W.STREAMINGLLM_480P, None, (3 + 4 + 3) * F),
            (W.DUMMY_FORCING_480P, (1 + 3) * F, (1 + 2 + 3) * F)]:
        w = w.with_(tokens_per_frame=F, n_heads=4, head_dim=16,
                    n_segments=6 if w.n_segments == 6 else F)
        hm = W.head_map(w)
        orc = O.ForcingKVOracle.from_workload(w, hm)
        hk, hv, ck, cv, q = W.snapshot_inputs(w)
        orc.append_frames(0, hk, hv)
        orc.set_current(0, ck, cv)
        for h in range(4):
            n = orc.view_length(0, h)
            assert n == (want_static if hm[0, h] else want_dynamic), (w.name, h, n)


# ---------------------------------------------------------------- FP8 attention (e4m3 Q K^T)
def _e4m3_codes():
    """Every finite OCP FP8 E4M3 value, decoded from its bit fields: sign, 4 exponent bits
    with bias 7 (0 = subnormal, m 2^-9), 3 mantissa bits; S.1111.111 is NaN."""
    vals = []
    for code in range(256):
        s, e, m = code >> 7, (code >> 3) & 15, code & 7
        if e == 15 and m == 7:
            continue
        v = m * 2.0 ** -9 if e == 0 else (1 + m / 8) * 2.0 ** (e - 7)
        vals.append(-v if s else v)
    return np.array(vals)


def test_e4m3_grid_round_trips():
    v = _e4m3_codes()
    assert v.max() == 448.0 and np.min(np.abs(v[v != 0])) == 2.0 ** -9
    assert np.array_equal(O.e4m3_round(v), v)


def test_e4m3_midpoints_round_to_even_mantissa():
    pos = np.unique(_e4m3_codes()[_e4m3_codes() >= 0])
    mid = (pos[:-1] + pos[1:]) / 2
    got = O.e4m3_round(mid)
    # the even neighbour: mantissa field (value / spacing) even in the neighbours' binade
    for lo, hi, g in zip(pos[:-1], pos[1:], got):
        spacing = hi - lo
        even = lo if round(lo / spacing) % 2 == 0 else hi
        assert g == even, (lo, hi, g)
    assert np.array_equal(O.e4m3_round(-mid), -got)


def test_e4m3_matches_torch_cast_on_every_bf16_in_range():
    bits = np.arange(1 << 16, dtype=np.uint32)
    f = (bits << 16).astype(np.uint32).view(np.float32)
    f = f[np.isfinite(f) & (np.abs(f) <= 448.0)]
    ref = torch.from_numpy(f).to(torch.float8_e4m3fn).float().numpy().astype(np.float64)
    assert np.array_equal(O.e4m3_round(f.astype(np.float64)), ref)


def test_e4m3_saturates():
    assert np.array_equal(O.e4m3_round([449.0, 464.0, 1e6, -500.0]), [448.0, 448.0, 448.0, -448.0])


def test_q_row_exponent_is_the_smallest_fitting_power():
    rng = np.random.default_rng(5)
    amax = np.concatenate([rng.lognormal(0, 6, 2000), [448.0, 449.0, 224.0, 896.0, 1.0, 2.0 ** -100]])
    for a in amax:
        e = O.q_row_exponent(a)
        assert a <= 448.0 * 2.0 ** e and a > 448.0 * 2.0 ** (e - 1), (a, e)
    assert (O.q_row_exponent(0.0), O.q_row_exponent(448.0), O.q_row_exponent(449.0),
            O.q_row_exponent(1.0)) == (0, 0, 1, -8)


def test_fp8_attention_is_exact_on_e4m3_inputs():
    # Q rows and K already on the (row-scaled) e4m3 grid: quantization changes nothing
    rng = np.random.default_rng(6)
    grid = _e4m3_codes()
    grid = grid[(np.abs(grid) >= 2.0 ** -3) & (np.abs(grid) <= 8)]
    Q = rng.choice(grid, size=(40, 64)) * np.ldexp(1.0, rng.integers(-3, 4, size=40))[:, None]
    K = rng.choice(grid, size=(300, 64))
    V = rng.standard_normal((300, 64))
    assert np.array_equal(O.attention_fp8_qk(Q, K, V), O.attention_fp64(Q, K, V))


def test_fp8_attention_quantizes_within_e4m3_error():
    rng = np.random.default_rng(7)
    Q = rng.standard_normal((64, 128)) * np.ldexp(1.0, rng.integers(-6, 1, size=64))[:, None]
    K = rng.standard_normal((500, 128))
    V = rng.standard_normal((500, 128))
    q8, e = O.quantize_q_rows(Q)
    deq = q8 * np.ldexp(1.0, e)[:, None]
    # relative rounding error of e4m3 normals <= 2^-4; every row uses the full range
    normal = np.abs(deq) >= 2.0 ** -6 * np.ldexp(1.0, e)[:, None]
    assert np.all(np.abs(deq - Q)[normal] <= np.abs(Q)[normal] * 2.0 ** -4 + 1e-300)
    assert np.all(np.abs(q8).max(axis=1) >= 224.0)   # amax 2^-e in (224, 448], then rounded
    ref, got = O.attention_fp64(Q, K, V), O.attention_fp8_qk(Q, K, V)
    assert 1e-5 < np.abs(got - ref).max() < 0.1


# ---- FP8 attention with P V on e4m3 operands too
def test_fp8_pv_one_key_returns_the_rounded_value():
    # a single key with logit 0: reference ceil(0) = 0, numerator 2^6 = 64 (on the grid), so
    # O = e4m3(V) exactly, whatever the query
    rng = _rng(41)
    Q, V = _bf16(rng.standard_normal((5, 128))), _bf16(rng.standard_normal((1, 128)) * 3)
    out = O.attention_fp8(Q, np.zeros((1, 128)), V)
    assert np.array_equal(out, np.repeat(O.e4m3_round(V), 5, axis=0))


def test_fp8_pv_reference_is_the_row_max_rounded_up():
    # one key, logit 2.75 / 8 = 0.34375 (q = 1 and k = 2.75 on channel 0, both e4m3-exact; the
    # query row scales to 256): y = 0.34375 / ln 2 = 0.496, reference ceil(y) = 1, numerator
    # n = 2^(y + 5) = 45.13, which rounds to 44 on the e4m3 grid (binade [32, 64), step 4);
    # O = 44 / n x e4m3(V).  With the exact row maximum as reference (n = 64) O would be e4m3(V).
    D = 64
    Q = np.zeros((1, D))
    Q[0, 0] = 1.0
    K = np.zeros((1, D))
    K[0, 0] = 2.75
    V = np.full((1, D), 3.0)
    n = 2.0 ** (0.34375 / math.log(2.0) + 5.0)
    assert 44.0 < n < 46.0
    out = O.attention_fp8(Q, K, V)
    assert np.allclose(out, 44.0 / n * 3.0, rtol=1e-14, atol=0)


def test_fp8_pv_equal_keys_average_the_rounded_values():
    # equal keys with logit 0: every numerator is 64 (exact), O = mean of e4m3(V)
    rng = _rng(42)
    Q = _bf16(rng.standard_normal((3, 64)))
    V = _bf16(rng.standard_normal((7, 64)))
    out = O.attention_fp8(Q, np.zeros((7, 64)), V)
    want = O.e4m3_round(V).mean(axis=0)
    assert np.abs(out - want[None, :]).max() <= 1e-15


def test_fp8_pv_scale_is_two_to_the_six():
    # two keys with logits 0 and -12 (q = 8 on channel 0, keys 0 and -12 there: all exact in
    # e4m3, the query row scaled by 2^5 to 256): reference 0, numerators 2^6 and 2^6 e^-12 =
    # 3.9e-4, below half the smallest e4m3 step (2^-10): it rounds to 0, so O = 0 exactly although
    # the second key's value is 448; a scale of 2^8 (or an unrounded numerator) would leave a
    # visible 448 e^-12 / (1 + e^-12) = 2.7e-3
    D = 64
    Q = np.zeros((1, D))
    Q[0, 0] = 8.0
    K = np.zeros((2, D))
    K[1, 0] = -12.0
    V = np.zeros((2, D))
    V[1, :] = 448.0
    out = O.attention_fp8(Q, K, V)
    assert np.array_equal(out, np.zeros((1, D)))
    assert np.allclose(O.attention_fp8_qk(Q, K, V), 448.0 * math.exp(-12) / (1 + math.exp(-12)),
                       rtol=1e-12, atol=0)
    # the first key alone: numerator 64 on the grid, weight 64 / (64 (1 + e^-12))
    V[0, :], V[1, :] = 2.0, 0.0
    assert np.allclose(O.attention_fp8(Q, K, V), 2.0 / (1 + math.exp(-12)), rtol=1e-14, atol=0)


def test_fp8_pv_within_the_e4m3_error_of_its_numerators():
    # against the same attention with unrounded numerators (fp8_qk on e4m3(V)): each numerator
    # x moves by at most max(2^-4 x, 2^-10) (half an e4m3 step)
    rng = _rng(43)
    D = 128
    Q = _bf16(rng.standard_normal((40, D)))
    K = _bf16(rng.standard_normal((300, D)) * 1.5)
    V = _bf16(rng.standard_normal((300, D)))
    got = O.attention_fp8(Q, K, V)
    ref = O.attention_fp8_qk(Q, K, O.e4m3_round(V))
    q8, e = O.quantize_q_rows(Q)
    y = (q8 * np.ldexp(1.0, e)[:, None]) @ O.e4m3_round(K).T / (math.sqrt(D) * math.log(2.0))
    x = np.exp2(y - np.ceil(y.max(axis=1, keepdims=True)) + 6)
    assert x.max() <= 64.0 and x.max(axis=1).min() > 32.0
    bound = (np.maximum(x * 2.0 ** -4, 2.0 ** -10) @ np.abs(O.e4m3_round(V))) / x.sum(axis=1, keepdims=True)
    assert (np.abs(got - ref) <= bound * (1 + 1e-9) + 1e-15).all()
    assert np.abs(got - ref).max() > 0                    # the rounding is not a no-op


def test_fp8_pv_power_of_two_reference_shift_changes_nothing():
    # scaling every numerator by 2^k (a kernel's running reference below the row's) leaves the
    # e4m3 rounding of normal values unchanged: numerators above 2^-6 for k in {0, 1, 2}
    rng = _rng(44)
    x = np.exp2(rng.uniform(-6.0, 6.0, 5000))
    for k in (1, 2):
        assert np.array_equal(O.e4m3_round(x * 2.0 ** k), O.e4m3_round(x) * 2.0 ** k)
