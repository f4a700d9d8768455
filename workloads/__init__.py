"""Seeded synthetic workloads for the Forcing-KV hot path.

This module holds the workload definitions (shapes, schedules and value models
shaped like the paper's 480P / 1080P Self Forcing and LongLive settings, Sec. 5
and App. H) and one counter-based random generator.  The CPU oracle and the
CUDA path are both fed from here, byte for byte.  Nothing in this module
computes any part of the method: no scores, no selection, no attention.

Generator (fixed recipe, independent of platform):
  * SplitMix64 (Steele, Lea & Flood, OOPSLA 2014) over a 64-bit counter,
  * Box-Muller in fp64 on the two 24-bit halves of each 64-bit draw,
  * fp64 -> fp32 (round to nearest) -> bf16 (round to nearest even).

Value model (per layer, per head, per token, per channel):
  * keys   K_f = s_h * x_f, x_f = rho_k * x_{f-1} + sqrt(1 - rho_k^2) * e_f,
    x_0 = e_0, and x_f = e_f at a scene-cut frame;  s_h ~ U[scale_lo, scale_hi];
  * values the same AR(1) recursion with rho_v and no head scale;
  * queries iid N(0, 1).
"""
from __future__ import annotations

import math
import os
from concurrent.futures import ThreadPoolExecutor
from dataclasses import dataclass, field, replace
from typing import Iterator

import numpy as np

__all__ = [
    "Workload", "TINY", "TINY_PER_FRAME", "P480_LAYER", "P480_STACK", "ROLLING",
    "P1080_LAYER", "WORKLOADS", "normals", "uniforms", "to_bf16_bits", "bf16_bits_to_f32",
    "profile_inputs", "FULL_KV_480P", "STREAMINGLLM_480P", "DUMMY_FORCING_480P", "UNIFORM_TOKENS_480P",
    "RANDOM_TOKENS_480P", "P480_LAYER_FP8PV", "P1080_LAYER_FP8PV", "TINY_FP8PV",
    "head_map", "FrameStream", "snapshot_inputs", "queries", "step_kv", "stream_key",
]

_U64 = np.uint64
_THREADS = max(1, min(16, os.cpu_count() or 1))


def _splitmix64(x: np.ndarray) -> np.ndarray:
    with np.errstate(over="ignore"):
        z = x + _U64(0x9E3779B97F4A7C15)
        z = (z ^ (z >> _U64(30))) * _U64(0xBF58476D1CE4E5B9)
        z = (z ^ (z >> _U64(27))) * _U64(0x94D049BB133111EB)
        return z ^ (z >> _U64(31))


def stream_key(*tags: int) -> int:
    """Fold integer tags (seed, tensor kind, layer, frame, ...) into one 64-bit key."""
    k = np.array([0x51ED2701F00DCAFE], dtype=np.uint64)
    for t in tags:
        with np.errstate(over="ignore"):
            k = _splitmix64(k ^ np.array([t & 0xFFFFFFFFFFFFFFFF], dtype=np.uint64))
    return int(k[0])


def normals(key: int, n: int) -> np.ndarray:
    """n standard normal draws (fp64) of stream `key`."""
    m = (n + 1) // 2
    with np.errstate(over="ignore"):
        z = _splitmix64(_U64(key) + np.arange(m, dtype=np.uint64))
    u1 = ((z >> _U64(40)).astype(np.float64) + 1.0) * (1.0 / 16777216.0)        # (0, 1]
    u2 = ((z >> _U64(16)) & _U64(0xFFFFFF)).astype(np.float64) * (1.0 / 16777216.0)  # [0, 1)
    r = np.sqrt(-2.0 * np.log(u1))
    out = np.empty(2 * m, dtype=np.float64)
    out[0::2] = r * np.cos(2.0 * math.pi * u2)
    out[1::2] = r * np.sin(2.0 * math.pi * u2)
    return out[:n]


def uniforms(key: int, n: int) -> np.ndarray:
    """n uniform draws in [0, 1) (fp64) of stream `key`."""
    with np.errstate(over="ignore"):
        z = _splitmix64(_U64(key) + np.arange(n, dtype=np.uint64))
    return (z >> _U64(11)).astype(np.float64) * (1.0 / 9007199254740992.0)


def to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """fp64/fp32 -> fp32 (nearest) -> bf16 bit pattern (nearest even), as uint16."""
    b = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
    with np.errstate(over="ignore"):
        r = (b + np.uint32(0x7FFF) + ((b >> np.uint32(16)) & np.uint32(1))) >> np.uint32(16)
    return r.astype(np.uint16)


def bf16_bits_to_f32(bits: np.ndarray) -> np.ndarray:
    """bf16 bit pattern (uint16) -> exact fp32 value."""
    return (np.asarray(bits, dtype=np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32)


# tensor-kind tags of the generator streams
_K, _V, _Q, _SCALE, _MAP, _KSTEP, _VSTEP = 1, 2, 3, 4, 5, 6, 7
_PK, _PQ, _PB, _PT = 11, 12, 13, 14   # head-profiling inputs


@dataclass(frozen=True)
class Workload:
    """One synthetic workload: cache/attention shapes plus its driving schedule.

    schedule "snapshot": `n_history_frames` frames are loaded as history, then one
    chunk of C frames is the current chunk (single-layer cases).
    schedule "stream": `n_chunks` chunks are appended one by one; after each append
    the cache is compressed and the chunk is attended `denoise_steps` times.
    """
    name: str
    n_layers: int
    n_heads: int
    head_dim: int
    tokens_per_frame: int
    frames_per_chunk: int
    n_sink_frames: int
    window_frames: int            # non-sink history frames kept (0 = unbounded)
    n_segments: int
    keep_budget_permille: int
    select_scope: str = "per_frame"      # "per_frame" | "pooled"
    score_source: str = "per_head"       # "per_head" | "layer0_pooled"
    incremental: bool = False
    schedule: str = "snapshot"
    n_history_frames: int = 0
    n_chunks: int = 0
    denoise_steps: int = 1
    rho_k: float = 0.9
    rho_v: float = 0.9
    scale_lo: float = 0.5
    scale_hi: float = 2.0
    scene_cut_every_chunks: int = 0
    static_heads: tuple = ()             # fixed static heads (empty = seeded map)
    static_fraction: float = 0.5
    exact_half_static: bool = True       # seeded permutation with exactly H/2 static
    selection: str = "similarity"        # "similarity" | "all" | "uniform" | "random"
    select_seed: int = 0
    static_drop_anchor: bool = False
    attn_precision: str = "bf16"         # "bf16" | "fp8_qk" (Q K^T on e4m3 operands) | "fp8" (P V too)
    seed: int = 0
    description: str = ""

    # ---- derived sizes ----
    @property
    def seg_len(self) -> int:
        return self.tokens_per_frame // self.n_segments

    @property
    def n_queries(self) -> int:
        return self.frames_per_chunk * self.tokens_per_frame

    def max_history_frames(self) -> int:
        if self.schedule == "snapshot":
            return self.n_history_frames
        return self.n_chunks * self.frames_per_chunk

    def scene_cut(self, frame: int) -> bool:
        e = self.scene_cut_every_chunks
        return e > 0 and frame > 0 and frame % (e * self.frames_per_chunk) == 0

    def with_(self, **kw) -> "Workload":
        return replace(self, **kw)


TINY = Workload(
    name="tiny", n_layers=1, n_heads=4, head_dim=64, tokens_per_frame=60, frames_per_chunk=3,
    n_sink_frames=0, window_frames=0, n_segments=1, keep_budget_permille=500,
    select_scope="pooled", schedule="snapshot", n_history_frames=7,
    rho_k=0.8, rho_v=0.0, scale_lo=1.0, scale_hi=1.0, static_heads=(0, 1), seed=0,
    description="tiny correctness case: 1 layer, 4 heads (0-1 static), D=64, 60 tokens/frame, "
                "3-frame chunk, 7 history frames, one segment per frame, 50% budget pooled")

TINY_PER_FRAME = TINY.with_(
    name="tiny_per_frame", n_segments=6, select_scope="per_frame",
    description="tiny case with 6 segments (grid rows) per frame, 3 of 6 kept per frame")

P480_LAYER = Workload(
    name="480p_layer", n_layers=1, n_heads=12, head_dim=128, tokens_per_frame=1560,
    frames_per_chunk=3, n_sink_frames=1, window_frames=0, n_segments=6, keep_budget_permille=700,
    schedule="snapshot", n_history_frames=19, seed=1,
    description="480P single layer: 12 heads (6 static seeded), D=128, 1560 tokens/frame (30x52), "
                "4680 queries, 1 sink + 18 history frames, 70% dynamic budget")

P480_STACK = Workload(
    name="480p_stack", n_layers=30, n_heads=12, head_dim=128, tokens_per_frame=1560,
    frames_per_chunk=3, n_sink_frames=1, window_frames=0, n_segments=6, keep_budget_permille=700,
    score_source="layer0_pooled", incremental=True, schedule="stream", n_chunks=7, denoise_steps=4,
    exact_half_static=False, seed=2,
    description="480P stack: 30 layers x 12 heads, 7 chunks of 3 frames, 4 denoising steps, "
                "compression after each append, layer-0 pooled scoring")

ROLLING = Workload(
    name="rolling", n_layers=1, n_heads=12, head_dim=128, tokens_per_frame=1560,
    frames_per_chunk=3, n_sink_frames=1, window_frames=12, n_segments=6, keep_budget_permille=600,
    incremental=True, schedule="stream", n_chunks=60, denoise_steps=1,
    rho_k=0.95, rho_v=0.95, scene_cut_every_chunks=20, seed=3,
    description="rolling cache: 12 heads, D=128, 1 sink + 12-frame window, 60 chunks, 60% budget, "
                "rho=0.95 drift with a scene cut every 20 chunks")

P1080_LAYER = Workload(
    name="1080p_layer", n_layers=1, n_heads=12, head_dim=128, tokens_per_frame=8160,
    frames_per_chunk=3, n_sink_frames=1, window_frames=0, n_segments=6, keep_budget_permille=700,
    schedule="snapshot", n_history_frames=10, seed=4,
    description="1080P single layer: 12 heads, D=128, 8160 tokens/frame (68x120), 24480 queries, "
                "1 sink + 9 history frames, 70% dynamic budget")

# The paper's comparison rules (App. H, Sec. 5.3) on the 480P layer snapshot, for speed
# comparisons through the same kernels (their quality claims need model weights).
FULL_KV_480P = P480_LAYER.with_(
    name="full_kv_480p", selection="all", exact_half_static=False, static_fraction=0.0,
    description="the uncompressed cache on the 480P layer: every head keeps every frame of the "
                "window (the paper's full-KV reference)")
STREAMINGLLM_480P = P480_LAYER.with_(
    name="streamingllm_480p", n_sink_frames=3, window_frames=4, selection="all",
    exact_half_static=False, static_fraction=0.0,
    description="frame-level StreamingLLM on the 480P layer: every head keeps 3 sink frames and "
                "the 4 most recent history frames")
DUMMY_FORCING_480P = P480_LAYER.with_(
    name="dummy_forcing_480p", window_frames=2, selection="all", static_drop_anchor=True,
    description="Dummy Forcing (L = 2) on the 480P layer: local heads keep the sink and the chunk, "
                "neighbour heads the sink and the last 2 history frames")
UNIFORM_TOKENS_480P = P480_LAYER.with_(
    name="uniform_tokens_480p", n_segments=1560, selection="uniform",
    description="uniform token pruning on the 480P layer's dynamic heads: 1092 evenly spaced "
                "tokens of each history frame (70%)")
RANDOM_TOKENS_480P = P480_LAYER.with_(
    name="random_tokens_480p", n_segments=1560, selection="random", select_seed=7,
    description="random token pruning on the 480P layer's dynamic heads: 1092 seeded random "
                "tokens of each history frame (70%)")

# FP8 attention on the compressed cache (the paper's quantization appendix): Q K^T on e4m3.
P480_LAYER_FP8 = P480_LAYER.with_(
    name="480p_layer_fp8", attn_precision="fp8_qk",
    description="the 480P layer with Q K^T on FP8 E4M3 operands (per-row power-of-two query "
                "scales, unscaled keys), P V in bf16")
P1080_LAYER_FP8 = P1080_LAYER.with_(
    name="1080p_layer_fp8", attn_precision="fp8_qk",
    description="the 1080P layer with Q K^T on FP8 E4M3 operands, P V in bf16")
TINY_FP8 = TINY_PER_FRAME.with_(
    name="tiny_fp8", head_dim=128, attn_precision="fp8_qk",
    description="tiny per-frame case at head_dim 128 with Q K^T on FP8 E4M3 operands")
# both products on e4m3 operands (P scaled by 2^6 relative to the running row max, V unscaled)
P480_LAYER_FP8PV = P480_LAYER.with_(
    name="480p_layer_fp8pv", attn_precision="fp8",
    description="the 480P layer with Q K^T and P V on FP8 E4M3 operands")
P1080_LAYER_FP8PV = P1080_LAYER.with_(
    name="1080p_layer_fp8pv", attn_precision="fp8",
    description="the 1080P layer with Q K^T and P V on FP8 E4M3 operands")
TINY_FP8PV = TINY_PER_FRAME.with_(
    name="tiny_fp8pv", head_dim=128, attn_precision="fp8",
    description="tiny per-frame case at head_dim 128 with both products on FP8 E4M3 operands")

WORKLOADS = {w.name: w for w in (TINY, TINY_PER_FRAME, P480_LAYER, P480_STACK, ROLLING, P1080_LAYER,
                                 FULL_KV_480P, STREAMINGLLM_480P, DUMMY_FORCING_480P,
                                 UNIFORM_TOKENS_480P, RANDOM_TOKENS_480P, P480_LAYER_FP8,
                                 P1080_LAYER_FP8, TINY_FP8, P480_LAYER_FP8PV, P1080_LAYER_FP8PV,
                                 TINY_FP8PV)}


def head_map(w: Workload) -> np.ndarray:
    """uint8 [n_layers, n_heads]: 1 = static head, 0 = dynamic head (seeded)."""
    m = np.zeros((w.n_layers, w.n_heads), dtype=np.uint8)
    for layer in range(w.n_layers):
        if w.static_heads:
            m[layer, list(w.static_heads)] = 1
        elif w.exact_half_static:
            u = uniforms(stream_key(w.seed, _MAP, layer), w.n_heads)
            m[layer, np.argsort(u, kind="stable")[: w.n_heads // 2]] = 1
        else:
            u = uniforms(stream_key(w.seed, _MAP, layer), w.n_heads)
            m[layer] = (u < w.static_fraction).astype(np.uint8)
    return m


def _head_scales(w: Workload, layer: int) -> np.ndarray:
    u = uniforms(stream_key(w.seed, _SCALE, layer), w.n_heads)
    return w.scale_lo + (w.scale_hi - w.scale_lo) * u


class FrameStream:
    """Sequential AR(1) key/value frames of one layer, as bf16 bits [F, H, D]."""

    def __init__(self, w: Workload, layer: int):
        self.w, self.layer, self.next = w, layer, 0
        self._xk = None
        self._xv = None
        self._scale = _head_scales(w, layer)[None, :, None]

    def _noise(self, kind, f):
        w = self.w
        e = normals(stream_key(w.seed, kind, self.layer, f),
                    w.tokens_per_frame * w.n_heads * w.head_dim)
        return e.reshape(w.tokens_per_frame, w.n_heads, w.head_dim)

    def _advance(self, x, rho, e, f):
        if x is None or self.w.scene_cut(f):
            return e
        return rho * x + math.sqrt(max(0.0, 1.0 - rho * rho)) * e

    def next_frame(self) -> tuple[np.ndarray, np.ndarray]:
        k, v = self.frames(1)
        return k, v

    def frames(self, n: int) -> tuple[np.ndarray, np.ndarray]:
        """The next n frames, concatenated token-major: [n*F, H, D] each."""
        w = self.w
        F = w.tokens_per_frame
        K = np.empty((n * F, w.n_heads, w.head_dim), np.uint16)
        V = np.empty((n * F, w.n_heads, w.head_dim), np.uint16)
        if n == 0:
            return K, V
        fs = list(range(self.next, self.next + n))
        jobs = [(_K, f) for f in fs] + [(_V, f) for f in fs]
        with ThreadPoolExecutor(max_workers=min(len(jobs), _THREADS)) as ex:
            noise = dict(zip(jobs, ex.map(lambda kf: self._noise(*kf), jobs)))
        for i, f in enumerate(fs):
            self._xk = self._advance(self._xk, w.rho_k, noise[(_K, f)], f)
            self._xv = self._advance(self._xv, w.rho_v, noise[(_V, f)], f)
            K[i * F:(i + 1) * F] = to_bf16_bits(self._scale * self._xk)
            V[i * F:(i + 1) * F] = to_bf16_bits(self._xv)
        self.next += n
        return K, V

    def chunks(self) -> Iterator[tuple[np.ndarray, np.ndarray]]:
        while True:
            yield self.frames(self.w.frames_per_chunk)


def snapshot_inputs(w: Workload, layer: int = 0):
    """(history K, history V [n_hist*F, H, D], current K, current V [C*F, H, D], Q [C*F, H, D])."""
    fs = FrameStream(w, layer)
    hk, hv = fs.frames(w.n_history_frames)
    ck, cv = fs.frames(w.frames_per_chunk)
    q = queries(w, layer, 0, 0)
    return hk, hv, ck, cv, q


def queries(w: Workload, layer: int, chunk: int, step: int) -> np.ndarray:
    """Queries of one chunk at one denoising step: iid N(0,1) bf16 bits [C*F, H, D]."""
    n = w.n_queries * w.n_heads * w.head_dim
    q = normals(stream_key(w.seed, _Q, layer, chunk, step), n)
    return to_bf16_bits(q).reshape(w.n_queries, w.n_heads, w.head_dim)


def step_kv(w: Workload, layer: int, chunk: int, step: int, clean_k: np.ndarray,
            clean_v: np.ndarray) -> tuple[np.ndarray, np.ndarray]:
    """Current-chunk K/V at denoising step `step`: the clean chunk on the last step,
    earlier steps add seeded noise of decreasing weight (a stand-in for noisy latents)."""
    last = w.denoise_steps - 1
    if step >= last:
        return clean_k, clean_v
    a = 0.5 * (last - step) / max(1, last)
    n = clean_k.size
    ek = normals(stream_key(w.seed, _KSTEP, layer, chunk, step), n).reshape(clean_k.shape)
    ev = normals(stream_key(w.seed, _VSTEP, layer, chunk, step), n).reshape(clean_v.shape)
    k = bf16_bits_to_f32(clean_k).astype(np.float64) + a * ek
    v = bf16_bits_to_f32(clean_v).astype(np.float64) + a * ev
    return to_bf16_bits(k), to_bf16_bits(v)


def profile_inputs(seed: int, n_heads: int, head_dim: int, tokens_per_frame: int,
                   frames_per_chunk: int, n_sink_frames: int, n_history_frames: int):
    """Seeded inputs of one offline head-profiling pass (one layer, one step).

    Keys of the attention window, token-major [Nk, H, D], in the order [generated chunk (C
    frames) | sink frames | other history | transition frame (the newest history frame)];
    queries [C*F, H, D] of the generated chunk.  Head h's queries are beta_h times the
    generated chunk's own keys plus unit noise (beta_h uniform in [0, 1.4)), and the
    transition frame's keys are 0.7 x the chunk's last frame plus 0.7 x noise, so that the
    heads range from attending locally to attending across the whole window.  Returns
    (Q bits, K bits, (n_generate, n_sink, n_transition)) as bf16 bit patterns."""
    F, C, S, H, D = tokens_per_frame, frames_per_chunk, n_sink_frames, n_heads, head_dim
    assert n_history_frames > S
    n_gen, n_sink, n_trans = C * F, S * F, F
    nk = n_gen + (n_history_frames - 1) * F + n_trans
    K = normals(stream_key(seed, _PK), nk * H * D).reshape(nk, H, D)
    K[nk - F:] = 0.7 * K[n_gen - F:n_gen] + 0.7 * normals(stream_key(seed, _PT), F * H * D).reshape(F, H, D)
    beta = 1.4 * uniforms(stream_key(seed, _PB), H)
    Q = beta[None, :, None] * K[:n_gen] + normals(stream_key(seed, _PQ), n_gen * H * D).reshape(n_gen, H, D)
    return to_bf16_bits(Q), to_bf16_bits(K), (n_gen, n_sink, n_trans)
