"""Second comparison of the score contract against the paper's definition (Sec. 4.3, Eq. 3).

The keep decision is taken on fp32 scores under the score contract (the kernel's precision);
the paper defines the score as the cosine of two key segments.  For every scored (t, j) of a
workload state this module compares the contract score with the fp64 cosine, and compares
BottomK on the contract scores with BottomK on the fp64 scores.  A kept-set difference can
only come from a near-tie: two candidates whose fp64 scores lie within twice the contract's
deviation of each other at the keep/evict boundary.  Oracle and workload generator only."""
from __future__ import annotations

import numpy as np

import oracle as O
import workloads as W

SCORE_FP64_TOL = 1e-6     # |contract - fp64| bound on unit-scale scores


def _boundary_gap(vals: np.ndarray, k: int) -> float:
    """fp64 gap between the k-th and (k+1)-th smallest values (inf when no boundary)."""
    if k <= 0 or k >= len(vals):
        return float("inf")
    s = np.sort(vals)
    return float(s[k] - s[k - 1])


def compare_state(orc: O.ForcingKVOracle, layer: int, heads) -> dict:
    """Contract vs fp64 scores and kept sets of the dynamic heads `heads` of `layer`."""
    n = orc.n
    out = {"scored": 0, "max_abs": 0.0, "disagree": 0, "unexplained": 0}
    for h in heads:
        sc = orc.scores(layer, h)
        ex = orc.scores(layer, h, exact=True)
        for t in sc:
            d = np.abs(sc[t].astype(np.float64) - ex[t])
            out["scored"] += d.size
            out["max_abs"] = max(out["max_abs"], float(d.max()))
        kc = set(orc.kept(layer, h))
        kx = set(orc.kept(layer, h, exact=True))
        diff = kc ^ kx
        out["disagree"] += len(diff) // 2      # each swap replaces one kept segment
        if not diff:
            continue
        if orc.scope == "per_frame":
            k = orc._k_frame()
            for t in sorted({i // n for i in diff}):
                if _boundary_gap(ex[t], k) > 2 * SCORE_FP64_TOL:
                    out["unexplained"] += 1
        else:
            vals = np.concatenate([ex[t] for t in sorted(ex)])
            if _boundary_gap(vals, len(kc)) > 2 * SCORE_FP64_TOL:
                out["unexplained"] += 1
    return out


def _merge(acc: dict, r: dict) -> dict:
    if not acc:
        return dict(r)
    return {"scored": acc["scored"] + r["scored"], "max_abs": max(acc["max_abs"], r["max_abs"]),
            "disagree": acc["disagree"] + r["disagree"],
            "unexplained": acc["unexplained"] + r["unexplained"]}


def snapshot_case(w: W.Workload) -> dict:
    hm = W.head_map(w)
    hk, hv, ck, cv, _q = W.snapshot_inputs(w)
    orc = O.ForcingKVOracle.from_workload(w, hm)
    orc.append_frames(0, hk, hv)
    orc.set_current(0, ck, cv)
    return compare_state(orc, 0, [h for h in range(w.n_heads) if not hm[0, h]])


def stream_case(w: W.Workload, compare_every: int) -> dict:
    """The states a GPU stream test compares: after the append of chunk c for c a multiple of
    `compare_every` and the last chunk.  History frames are the clean frames (the last
    denoising step's K/V is the clean chunk)."""
    hm = W.head_map(w)
    orc = O.ForcingKVOracle.from_workload(w, hm, track_layers=[0])
    fs = W.FrameStream(w, 0)
    pooled = w.score_source == "layer0_pooled"
    # under layer-0 pooled scoring one kept set is shared: compare it once (head = any dynamic)
    dyn = [h for h in range(w.n_heads) if not hm[0, h]]
    heads = dyn[:1] if pooled else dyn
    acc: dict = {}
    for c in range(w.n_chunks):
        orc.append_chunk(0, *fs.frames(w.frames_per_chunk))
        if c % compare_every == 0 or c == w.n_chunks - 1:
            acc = _merge(acc, compare_state(orc, 0, heads))
    return acc


# the workload states of the GPU parity tests: name -> how to reach them
CASES = {
    "tiny": lambda: snapshot_case(W.TINY),
    "tiny_per_frame": lambda: snapshot_case(W.TINY_PER_FRAME),
    "480p_layer": lambda: snapshot_case(W.P480_LAYER),
    "1080p_layer": lambda: snapshot_case(W.P1080_LAYER),
    "rolling": lambda: stream_case(W.ROLLING, 10),
    "480p_stack": lambda: stream_case(W.P480_STACK, 3),
}
