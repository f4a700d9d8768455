"""Shared helpers of the GPU parity tests: drive the library and the oracle with the same
seeded inputs and compare kept sets (bit-exact), scores (bit-exact under the score contract;
tests/test_contract_vs_fp64.py compares the contract with the fp64 cosine on the same workload
states) and attention outputs (max abs <= 2e-2, mean abs <= 2e-3)."""
from __future__ import annotations

import functools

import numpy as np

import oracle as O
import workloads as W

ATOL_MAX = 2e-2      # attention tolerance vs the fp64 oracle (unit-variance bf16 inputs)
ATOL_MEAN = 2e-3


def to_dev(a: np.ndarray):
    import torch
    return torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).view(torch.bfloat16).cuda()


def to_f64(t) -> np.ndarray:
    import torch
    return t.detach().float().cpu().numpy().astype(np.float64)


@functools.lru_cache(maxsize=4)
def snapshot(w: W.Workload):
    return W.snapshot_inputs(w)


def sample_rows(nq: int, n: int = 96, seed: int = 0) -> np.ndarray:
    """Sampled query rows: random rows plus both ends of every boundary tile and the ragged tail."""
    rng = np.random.default_rng(seed)
    rows = set(rng.choice(nq, size=min(n, nq), replace=False).tolist())
    rows |= {0, min(127, nq - 1), min(128, nq - 1), nq - 1, max(0, nq - 2), (nq - 1) // 128 * 128}
    return np.array(sorted(rows))


def compare_layer(cache, orc, layer, Q_bits, O_dev, rows=None, heads=None, check_scores=True,
                  label=""):
    """Compare kept sets, scores, key counts and attention of one layer; returns stats."""
    H = orc.H
    heads = range(H) if heads is None else heads
    stats = {}
    for h in heads:
        assert cache.key_count(layer, h) == orc.view_length(layer, h), (label, layer, h)
        if orc.static[layer, h]:
            assert cache.kept(layer, h) == []
            continue
        kept_ref = orc.kept(layer, h)
        assert cache.kept(layer, h) == kept_ref, (label, layer, h)
        if check_scores:
            first, sc = cache.scores(layer, h)
            ref = orc.scores(layer, h)
            ts = sorted(ref)
            assert sc.shape[0] == len(ts), (label, layer, h)
            if ts:
                assert first == ts[0]
                ref_arr = np.stack([ref[t] for t in ts]).astype(np.float32)
                assert np.array_equal(sc.view(np.uint32), ref_arr.view(np.uint32)), (label, layer, h)
    nq = Q_bits.shape[0]
    rows = np.arange(nq) if rows is None else rows
    ref = orc.attend(layer, Q_bits, heads=list(heads), rows=rows)
    got = to_f64(O_dev)[rows]
    err = np.abs(got[:, list(heads)] - ref[:, list(heads)])
    stats["max_abs"] = float(err.max())
    stats["mean_abs"] = float(err.mean())
    assert np.isfinite(got[:, list(heads)]).all(), label
    assert stats["max_abs"] <= ATOL_MAX, (label, stats)
    assert stats["mean_abs"] <= ATOL_MEAN, (label, stats)
    return stats


def run_snapshot(w: W.Workload, rows=None, check_scores=True, inputs=None, head_map=None,
                 full_heads=None, **cache_over):
    """Load a snapshot workload into the library and the oracle, compress, attend, compare
    (`rows` of every head, then every row of the heads in `full_heads`)."""
    import torch
    from paper_2605_09681_gb300 import ForcingKVCache
    hk, hv, ck, cv, q = inputs if inputs is not None else snapshot(w)
    hm = W.head_map(w) if head_map is None else head_map
    with ForcingKVCache.from_workload(w, hm, **cache_over) as cache:
        cache.append_frames(0, to_dev(hk), to_dev(hv))
        cache.set_current(0, to_dev(ck), to_dev(cv))
        cache.compress()
        Od = cache.attend(0, to_dev(q))
        torch.cuda.synchronize()
        assert cache.sync_status() == 0
        orc = O.ForcingKVOracle.from_workload(w, hm)
        orc.append_frames(0, hk, hv)
        orc.set_current(0, ck, cv)
        st = compare_layer(cache, orc, 0, q, Od, rows=rows, check_scores=check_scores, label=w.name)
        if full_heads:
            full = compare_layer(cache, orc, 0, q, Od, heads=list(full_heads), check_scores=False,
                                 label=w.name + " every row")
            st["full_heads"] = list(full_heads)
            st["full_max_abs"], st["full_mean_abs"] = full["max_abs"], full["mean_abs"]
        return st


def run_stream(w, track_layers=(0,), compare_every=1, step_filter=None, layer_data=None):
    """Drive a streaming workload through the library and the oracle; compare tracked layers
    (every `compare_every` chunks and the last; denoising steps in `step_filter`, or all)."""
    import torch
    from paper_2605_09681_gb300 import ForcingKVCache
    hm = W.head_map(w)
    orc = O.ForcingKVOracle.from_workload(w, hm, track_layers=list(track_layers))
    streams = {l: W.FrameStream(w, l) for l in orc.layers}
    n_cmp = 0
    with ForcingKVCache.from_workload(w, hm) as cache:
        for c in range(w.n_chunks):
            clean = {l: streams[l].frames(w.frames_per_chunk) for l in orc.layers}
            for d in range(w.denoise_steps):
                kv = {l: W.step_kv(w, l, c, d, *clean[l]) for l in orc.layers}
                dev = {l: (to_dev(kv[l][0]), to_dev(kv[l][1])) for l in orc.layers}
                for l in range(w.n_layers):
                    src = l if l in dev else orc.layers[0]
                    if d == 0:
                        cache.append_chunk(l, *dev[src])
                    else:
                        cache.set_current(l, *dev[src])
                for l in orc.layers:
                    (orc.append_chunk if d == 0 else orc.set_current)(l, *kv[l])
                if d == 0:
                    cache.compress()
                check = (c % compare_every == 0 or c == w.n_chunks - 1) and (
                    step_filter is None or d in step_filter)
                for l in orc.layers:
                    q = W.queries(w, l, c, d)
                    Od = cache.attend(l, to_dev(q))
                    if check:
                        torch.cuda.synchronize()
                        rows = sample_rows(q.shape[0], 48, seed=c) if q.shape[0] > 1024 else None
                        compare_layer(cache, orc, l, q, Od, rows=rows, label="%s c%d d%d" % (w.name, c, d))
                        n_cmp += 1
        assert cache.sync_status() == 0
    return n_cmp
