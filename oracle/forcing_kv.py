"""CPU oracle of the Forcing-KV hot path (test infrastructure only).

This module is a plain, slow restatement of what the paper defines for one
chunk of autoregressive generation: the static-head key set (Sec. 4.2, Eq. 2),
segment-wise cosine scoring and BottomK selection for dynamic heads (Sec. 4.3,
Eq. 3), the dynamic-head key set (Sec. 4.3, Eq. 4) and softmax attention of the
chunk's queries over those keys.  Only the test suite, the smoke check and the
benchmark's CPU-baseline leg import it; the library never does, and it shares
no code with the CUDA path.

Floating point:
  * attention runs in fp64 on the exact bf16 input values;
  * every cosine is available in fp64 (`cosine_fp64`), the mathematical definition;
  * the keep/evict decision is an integer result decided by floating point, so it
    is taken in the kernel's precision, the "score contract" below, which both
    sides implement from its written definition:
      1. per token p, the channel dot d_p = sum_c a_c*b_c in fp32: channel group
         g (channels 8g..8g+7) is an fma chain from 0 in channel order; the D/8
         group partials are then combined by the butterfly p[g] += p[g ^ s] for
         s = D/16, ..., 2, 1 (fp32 adds) and p[0] is the result;
      2. each d_p is scaled by 2^24 (exact) and truncated toward zero to int64;
         the int64 values are summed over the segment's tokens (order-free);
      3. s = fp32( fp64(Dsum) / sqrt( fp64(N1) * fp64(N2) ) ), IEEE double with
         correct rounding; s = 0 when N1 == 0 or N2 == 0.
    Precondition: every token's contract squared norm n_p <= 2^23, which bounds
    every int64 partial by 2^47 and every sum by 2^63.

Readings taken where the paper is silent (each is listed with its reason in the
design notes): k = floor(b * n) segments kept per frame with b = 1 - r the keep
budget; cosine of two segments = Frobenius cosine of the flattened (F/n) x D key
blocks; the anchor frame is kept whole for dynamic heads and never scored; sink
frames are never scored and never evicted; a head profiled with all of its mass on the
sink frames is static (Eq. 1 has a zero denominator there); the window W counts non-sink history
frames including the anchor; ties in BottomK go to the lower index; the layer-0
proxy pools the int64 sums over all heads of layer 0.

Frames are numbered globally from 0 in append order; token p of frame f has the
global key id f*F + p; the current chunk is frames nh .. nh+C-1 where nh is the
number of history frames.
"""
from __future__ import annotations

from dataclasses import dataclass

import numpy as np

TWO24 = np.float32(16777216.0)
NORM_LIMIT = np.float32(8388608.0)  # 2^23, the scoring precondition on n_p


# --------------------------------------------------------------------------------------
# frame bookkeeping: Sec. 4.2 (Eq. 2: sink frames, anchor frame iC-1, current chunk),
# Sec. 4.3 (a history frame t is compared with t+1), App. H (sink preserved;
# compression starts at the second AR step, when adjacent history exists)
# --------------------------------------------------------------------------------------
@dataclass(frozen=True)
class FrameRoles:
    sink: tuple          # sink frames present in history
    window: tuple        # non-sink history frames inside the window (ascending)
    anchor: int | None   # transition-anchor frame (newest non-sink history frame)
    scoreable: tuple     # window frames t whose next frame t+1 is also in the window


def frame_roles(n_hist: int, n_sink: int, window: int) -> FrameRoles:
    """Roles of the history frames 0..n_hist-1 at one AR step (Eq. 2, Eq. 3)."""
    sink = tuple(range(min(n_sink, n_hist)))
    lo = n_sink if window <= 0 else max(n_sink, n_hist - window)
    win = tuple(range(lo, n_hist))
    anchor = win[-1] if win else None
    scoreable = win[:-1]
    return FrameRoles(sink, win, anchor, scoreable)


def segment_range(tokens_per_frame: int, n_segments: int, j: int) -> tuple[int, int]:
    """Token range of segment j: n contiguous equal parts of the frame (Sec. 4.3, App. H)."""
    if tokens_per_frame % n_segments:
        raise ValueError("tokens_per_frame must be a multiple of n_segments")
    L = tokens_per_frame // n_segments
    return j * L, (j + 1) * L


def keep_count(budget_permille: int, n_candidates: int) -> int:
    """floor(b * m) with b = budget_permille / 1000, in exact integer arithmetic (Eq. 3)."""
    return (budget_permille * n_candidates) // 1000


# --------------------------------------------------------------------------------------
# Eq. 3: segment cosine similarity
# --------------------------------------------------------------------------------------
def cosine_fp64(a: np.ndarray, b: np.ndarray) -> float:
    """Cosine of two key segments, flattened over tokens (and heads) and channels, fp64."""
    a = np.asarray(a, dtype=np.float64).ravel()
    b = np.asarray(b, dtype=np.float64).ravel()
    na, nb = float(a @ a), float(b @ b)
    if na == 0.0 or nb == 0.0:
        return 0.0
    return float((a @ b) / np.sqrt(na * nb))


def fmaf_bf16(a: np.ndarray, b: np.ndarray, c: np.ndarray) -> np.ndarray:
    """fp32 fused multiply-add a*b + c for bf16-valued a, b and fp32 c.

    a*b of two bf16 values has at most 16 significant bits, so it is exact in
    fp64; rounding (a*b + c) first to fp64 and then to fp32 equals a single
    rounding to fp32 for such operands (an operand too small to be exact in the
    fp64 sum lies below half an fp32 ulp of the other).
    """
    s = a.astype(np.float64) * b.astype(np.float64) + c.astype(np.float64)
    return s.astype(np.float32)


def token_dots_contract(A: np.ndarray, B: np.ndarray) -> np.ndarray:
    """Per-token channel dot in the contract's fp32 order. A, B: [T, D] fp32 (bf16 values)."""
    T, D = A.shape
    if D % 8:
        raise ValueError("head_dim must be a multiple of 8")
    G = D // 8
    Ag = A.reshape(T, G, 8)
    Bg = B.reshape(T, G, 8)
    acc = np.zeros((T, G), dtype=np.float32)
    for c in range(8):
        acc = fmaf_bf16(Ag[:, :, c], Bg[:, :, c], acc)
    s = G // 2
    idx = np.arange(G)
    while s >= 1:
        acc = (acc + acc[:, idx ^ s]).astype(np.float32)
        s //= 2
    return acc[:, 0]


def fixed_point(d: np.ndarray) -> np.ndarray:
    """trunc(d * 2^24) as int64 (the scaling is exact in fp32)."""
    return (np.asarray(d, dtype=np.float32) * TWO24).astype(np.int64)


def score_from_sums(dsum: int, n1: int, n2: int) -> np.float32:
    if n1 == 0 or n2 == 0:
        return np.float32(0.0)
    return np.float32(np.float64(dsum) / np.sqrt(np.float64(n1) * np.float64(n2)))


def segment_sums_contract(a: np.ndarray, b: np.ndarray) -> tuple[int, int, int]:
    """(Dsum, N1, N2) int64 sums of one segment pair under the contract.

    a, b: [..., T, D] fp32 arrays of bf16 values (a leading head axis is pooled)."""
    D = a.shape[-1]
    a2 = a.reshape(-1, D)
    b2 = b.reshape(-1, D)
    n1 = token_dots_contract(a2, a2)
    n2 = token_dots_contract(b2, b2)
    if (n1 > NORM_LIMIT).any() or (n2 > NORM_LIMIT).any():
        raise ValueError("scoring precondition violated: a token's squared key norm exceeds 2^23")
    d = token_dots_contract(a2, b2)
    with np.errstate(over="raise"):
        return (int(fixed_point(d).sum()), int(fixed_point(n1).sum()), int(fixed_point(n2).sum()))


def segment_score_contract(a: np.ndarray, b: np.ndarray) -> np.float32:
    """s_t^(j) of Eq. 3 under the score contract."""
    return score_from_sums(*segment_sums_contract(a, b))


# --------------------------------------------------------------------------------------
# Eq. 3: BottomK (keep the lowest-similarity segments, ties to the lower index)
# --------------------------------------------------------------------------------------
def bottom_k(scores, indices, k: int) -> list:
    """The k candidates with the smallest (score, index); returned in ascending index order."""
    order = sorted(zip((float(s) for s in scores), indices))
    return sorted(i for _, i in order[:k])


# --------------------------------------------------------------------------------------
# Eq. 2 and Eq. 4: key sets of a static and a dynamic head
# --------------------------------------------------------------------------------------
def frame_tokens(frame: int, F: int) -> list:
    return list(range(frame * F, (frame + 1) * F))


def static_key_tokens(roles: FrameRoles, F: int, current_frames, keep_anchor: bool = True) -> list:
    """Eq. 2: [sink frames, transition-anchor frame, current chunk] as global key ids
    (keep_anchor=False: sink and current chunk only, Dummy Forcing's local heads)."""
    ids = []
    for f in roles.sink:
        ids += frame_tokens(f, F)
    if roles.anchor is not None and keep_anchor:
        ids += frame_tokens(roles.anchor, F)
    for f in current_frames:
        ids += frame_tokens(f, F)
    return ids


def dynamic_key_tokens(roles: FrameRoles, F: int, n_segments: int, kept: list,
                       current_frames) -> list:
    """Eq. 4 plus the anchor frame: [sink, kept segments (t, j ascending), anchor, current].

    `kept` holds segment ids t*n + j.  The anchor is kept whole: a dynamic head's cache
    holds everything a static head keeps (Sec. 5.3, head-profiling ablation)."""
    ids = []
    for f in roles.sink:
        ids += frame_tokens(f, F)
    for sid in kept:
        t, j = divmod(sid, n_segments)
        lo, hi = segment_range(F, n_segments, j)
        ids += list(range(t * F + lo, t * F + hi))
    if roles.anchor is not None:
        ids += frame_tokens(roles.anchor, F)
    for f in current_frames:
        ids += frame_tokens(f, F)
    return ids


# --------------------------------------------------------------------------------------
# attention (Eq. 2 / Eq. 4 "Attention"): softmax(Q K^T / sqrt(D)) V in fp64
# --------------------------------------------------------------------------------------
def attention_fp64(Q: np.ndarray, K: np.ndarray, V: np.ndarray, row_block: int = 256) -> np.ndarray:
    """Textbook scaled dot-product attention, no mask. Q [Nq, D], K/V [Nk, D] -> [Nq, D]."""
    Q = np.asarray(Q, dtype=np.float64)
    K = np.asarray(K, dtype=np.float64)
    V = np.asarray(V, dtype=np.float64)
    scale = 1.0 / np.sqrt(Q.shape[1])
    out = np.empty((Q.shape[0], V.shape[1]), dtype=np.float64)
    for r0 in range(0, Q.shape[0], row_block):
        logits = (Q[r0:r0 + row_block] @ K.T) * scale
        logits -= logits.max(axis=1, keepdims=True)
        p = np.exp(logits)
        out[r0:r0 + row_block] = (p @ V) / p.sum(axis=1, keepdims=True)
    return out


# --------------------------------------------------------------------------------------
# FP8 attention (App. on quantization: FP8 attention on the compressed cache).  The paper
# names the technique only; the reading taken here: Q K^T on OCP FP8 E4M3 operands, P V
# unquantised.  K is rounded to e4m3 unscaled (e4m3's relative precision is the same over
# its normal range 2^-6..448; elements beyond 448 saturate); each query row (token, head) is scaled
# by a power of two 2^-e, e the smallest integer with max|q| <= 448 * 2^e, so scaling and
# unscaling are exact and the only rounding is the e4m3 rounding itself.
# --------------------------------------------------------------------------------------
E4M3_MAX = 448.0
E4M3_MIN_EXP = -6            # smallest normal binade 2^-6; subnormals step by 2^-9
E4M3_MANT_BITS = 3


def e4m3_round(x) -> np.ndarray:
    """Nearest OCP FP8 E4M3 value of each element (ties to the even mantissa), saturating
    to +-448; fp64 in, fp64 out.  The grid spacing in binade [2^b, 2^(b+1)) is
    2^(max(b, -6) - 3)."""
    x = np.asarray(x, dtype=np.float64)
    a = np.abs(x)
    _, ex = np.frexp(a)                          # a = m 2^ex, 0.5 <= m < 1: binade b = ex - 1
    b = np.maximum(ex.astype(np.int64) - 1, E4M3_MIN_EXP)
    spacing = np.ldexp(1.0, b - E4M3_MANT_BITS)
    r = np.rint(a / spacing) * spacing           # a / spacing is exact; rint ties to even
    r = np.minimum(r, E4M3_MAX)
    return np.copysign(r, x)


def q_row_exponent(amax: float) -> int:
    """Smallest integer e with amax <= 448 * 2^e (0 for amax = 0), clamped to [-120, 120]."""
    amax = float(amax)
    if amax == 0.0:
        return 0
    m, ex = np.frexp(amax)                       # amax = m 2^ex; 448 = 0.875 * 2^9
    e = int(ex) - 9 if m <= 0.875 else int(ex) - 8
    return max(-120, min(120, e))


def quantize_q_rows(Q: np.ndarray) -> tuple[np.ndarray, np.ndarray]:
    """Per-row FP8 quantization of queries: (e4m3 values of Q_r 2^-e_r as fp64, e_r)."""
    Q = np.asarray(Q, dtype=np.float64)
    e = np.array([q_row_exponent(np.abs(r).max()) if r.size else 0 for r in Q], dtype=np.int64)
    return e4m3_round(Q * np.ldexp(1.0, -e)[:, None]), e


def attention_fp8_qk(Q: np.ndarray, K: np.ndarray, V: np.ndarray) -> np.ndarray:
    """FP8 attention: softmax(2^e_r (Q8_r . K8) / sqrt(D)) V in fp64, with Q8, e from
    `quantize_q_rows`, K8 = e4m3_round(K) and V as given."""
    q8, e = quantize_q_rows(Q)
    return attention_fp64(q8 * np.ldexp(1.0, e)[:, None], e4m3_round(K), V)


# FP8 attention with P V on E4M3 operands too (the reading of the quantization appendix that
# also quantizes the value path): Q K^T exactly as in `attention_fp8_qk`; with each row's
# logits in log2 units, y_k = l_k / ln 2, and the row's reference R = ceil(max_k y_k) (the row
# maximum rounded up to an integer), the softmax numerators are n_k = 2^(y_k - R + 6), rounded
# to e4m3; V is rounded to e4m3 unscaled; the row's normaliser is the sum of the unrounded
# numerators:
#   O = sum_k e4m3(n_k) e4m3(V_k) / sum_k n_k.
# The numerators lie in (0, 2^6] (e4m3 max 448), with relative precision 2^-4 down to 2^-6 and
# subnormal steps of 2^-9 below.  An integer reference makes the rounding independent of where
# a kernel's running reference stands: two integer references differ by an exact power of two,
# under which e4m3 rounding of normal values is invariant.
P_SCALE_EXP = 6


def attention_fp8(Q: np.ndarray, K: np.ndarray, V: np.ndarray, row_block: int = 256) -> np.ndarray:
    """FP8 attention with both products on e4m3 operands, in fp64 on the rounded values."""
    q8, e = quantize_q_rows(Q)
    Qs = q8 * np.ldexp(1.0, e)[:, None]
    K8 = e4m3_round(K)
    V8 = e4m3_round(V)
    scale = 1.0 / (np.sqrt(Qs.shape[1]) * np.log(2.0))     # logits in log2 units
    out = np.empty((Qs.shape[0], V8.shape[1]), dtype=np.float64)
    for r0 in range(0, Qs.shape[0], row_block):
        y = (Qs[r0:r0 + row_block] @ K8.T) * scale
        R = np.ceil(y.max(axis=1, keepdims=True))
        n = np.exp2(y - R + P_SCALE_EXP)
        out[r0:r0 + row_block] = (e4m3_round(n) @ V8) / n.sum(axis=1, keepdims=True)
    return out


# --------------------------------------------------------------------------------------
# comparison selection rules (App. H, Sec. 5.3): ranking values replacing the scores
# --------------------------------------------------------------------------------------
_M64 = (1 << 64) - 1


def splitmix64(z: int) -> int:
    """SplitMix64 (Steele, Lea and Flood, 2014): the finaliser applied to z + golden gamma."""
    z = (z + 0x9E3779B97F4A7C15) & _M64
    z = ((z ^ (z >> 30)) * 0xBF58476D1CE4E5B9) & _M64
    z = ((z ^ (z >> 27)) * 0x94D049BB133111EB) & _M64
    return z ^ (z >> 31)


def rule_value(rule: str, seed: int, t: int, j: int, n: int, k: int) -> float:
    """Value of segment j of frame t under a comparison rule; BottomK keeps the smallest.
    all: 0 everywhere (k = n keeps every segment); uniform: 0 on the k evenly spaced segments
    {floor(i n / k) : i < k}, else 1; random: the top 24 bits of
    SplitMix64(seed * 2^40 xor t * 2^20 xor j) as a fraction of 2^24."""
    if rule == "all":
        return 0.0
    if rule == "uniform":
        return 0.0 if k > 0 and j in {i * n // k for i in range(k)} else 1.0
    if rule == "random":
        key = ((seed << 40) ^ (t << 20) ^ j) & _M64
        return (splitmix64(key) >> 40) / 16777216.0
    raise ValueError(rule)


# --------------------------------------------------------------------------------------
# offline head profiling (Sec. 4.1, Eq. 1)
# --------------------------------------------------------------------------------------
def head_attention_mass(Q: np.ndarray, K: np.ndarray, n_generate: int, n_sink: int,
                        n_transition: int, row_block: int = 256) -> np.ndarray:
    """Attention mass of one head per key class (Sec. 4.1), in fp64.

    Q [Nq, D], K [Nk, D] with the keys ordered [generated chunk | sink frames | other
    history | transition frame].  Each query row's softmax over all Nk keys (scale
    1/sqrt(D)) is summed per class and the rows are summed: returns
    [A_Total, A_Generate, A_Transition, A_Sink], where A_Total = sum over rows of the whole
    window's mass (each row contributes 1)."""
    Q = np.asarray(Q, dtype=np.float64)
    K = np.asarray(K, dtype=np.float64)
    nk = K.shape[0]
    assert n_generate + n_sink + n_transition <= nk
    scale = 1.0 / np.sqrt(Q.shape[1])
    gen = slice(0, n_generate)
    sink = slice(n_generate, n_generate + n_sink)
    trans = slice(nk - n_transition, nk)
    total = a_gen = a_trans = a_sink = 0.0
    for r0 in range(0, Q.shape[0], row_block):
        logits = (Q[r0:r0 + row_block] @ K.T) * scale
        logits -= logits.max(axis=1, keepdims=True)
        p = np.exp(logits)
        p /= p.sum(axis=1, keepdims=True)
        total += float(p.sum())
        a_gen += float(p[:, gen].sum())
        a_trans += float(p[:, trans].sum()) if n_transition else 0.0
        a_sink += float(p[:, sink].sum())
    return np.array([total, a_gen, a_trans, a_sink], dtype=np.float64)


def classify_head(mass, alpha: float) -> bool:
    """Eq. 1: static when (A_Generate + A_Transition) / (A_Total - A_Sink) > alpha.  A head
    whose whole mass is on the sink frames (denominator <= 0) is read as static."""
    total, a_gen, a_trans, a_sink = (float(x) for x in mass)
    window = total - a_sink
    if window <= 0.0:
        return True
    return (a_gen + a_trans) / window > alpha


# --------------------------------------------------------------------------------------
# streaming state: one AR generation, chunk by chunk
# --------------------------------------------------------------------------------------
def _bf16_to_f32(bits: np.ndarray) -> np.ndarray:
    return (np.asarray(bits, dtype=np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32)


class ForcingKVOracle:
    """Cache state of the method for a set of tracked layers.

    Inputs are bf16 bit patterns (uint16) laid out [tokens, heads, head_dim].  History
    frames outside the window (and not sinks) are dropped, as no later step reads them.
    """

    def __init__(self, *, n_layers, n_heads, head_dim, tokens_per_frame, frames_per_chunk,
                 n_sink_frames, window_frames, n_segments, keep_budget_permille,
                 select_scope="per_frame", score_source="per_head", head_is_static,
                 track_layers=None, selection="similarity", select_seed=0,
                 static_drop_anchor=False, attn_precision="bf16"):
        self.L, self.H, self.D = n_layers, n_heads, head_dim
        self.F, self.C = tokens_per_frame, frames_per_chunk
        self.S, self.W = n_sink_frames, window_frames
        self.n, self.b = n_segments, keep_budget_permille
        if tokens_per_frame % n_segments:
            raise ValueError("tokens_per_frame must be a multiple of n_segments")
        if select_scope not in ("per_frame", "pooled"):
            raise ValueError(select_scope)
        if score_source not in ("per_head", "layer0_pooled"):
            raise ValueError(score_source)
        self.scope, self.source = select_scope, score_source
        if selection not in ("similarity", "all", "uniform", "random"):
            raise ValueError(selection)
        self.selection, self.seed = selection, int(select_seed) & 0xFFFFFFFF
        self.keep_anchor_static = not static_drop_anchor
        if attn_precision not in ("bf16", "fp8_qk", "fp8"):
            raise ValueError(attn_precision)
        self.attn_precision = attn_precision
        self.static = np.asarray(head_is_static, dtype=np.uint8).reshape(n_layers, n_heads)
        self.layers = list(range(n_layers)) if track_layers is None else sorted(track_layers)
        if score_source == "layer0_pooled" and 0 not in self.layers:
            self.layers = [0] + self.layers
        self.nh = {l: 0 for l in self.layers}           # history frames appended
        self.frames = {l: {} for l in self.layers}      # frame -> (K [F,H,D] f32, V)
        self.current = {l: None for l in self.layers}   # (K [CF,H,D] f32, V)

    # ---- cache updates ----
    @classmethod
    def from_workload(cls, w, head_is_static, track_layers=None):
        return cls(n_layers=w.n_layers, n_heads=w.n_heads, head_dim=w.head_dim,
                   tokens_per_frame=w.tokens_per_frame, frames_per_chunk=w.frames_per_chunk,
                   n_sink_frames=w.n_sink_frames, window_frames=w.window_frames,
                   n_segments=w.n_segments, keep_budget_permille=w.keep_budget_permille,
                   select_scope=w.select_scope, score_source=w.score_source,
                   head_is_static=head_is_static, track_layers=track_layers,
                   selection=w.selection, select_seed=w.select_seed,
                   static_drop_anchor=w.static_drop_anchor, attn_precision=w.attn_precision)

    def _push_history(self, layer, K, V):
        F = self.F
        nf = K.shape[0] // F
        for i in range(nf):
            self.frames[layer][self.nh[layer]] = (K[i * F:(i + 1) * F], V[i * F:(i + 1) * F])
            self.nh[layer] += 1
        roles = frame_roles(self.nh[layer], self.S, self.W)
        live = set(roles.sink) | set(roles.window)
        for f in list(self.frames[layer]):
            if f not in live:
                del self.frames[layer][f]

    def append_frames(self, layer, K_bits, V_bits):
        """Append frames to history directly (the current chunk, if any, goes first)."""
        if layer not in self.nh:
            return
        if self.current[layer] is not None:
            self._push_history(layer, *self.current[layer])
            self.current[layer] = None
        self._push_history(layer, _bf16_to_f32(K_bits), _bf16_to_f32(V_bits))

    def append_chunk(self, layer, K_bits, V_bits):
        """The current chunk joins history; the new chunk becomes current."""
        if layer not in self.nh:
            return
        if self.current[layer] is not None:
            self._push_history(layer, *self.current[layer])
        self.current[layer] = (_bf16_to_f32(K_bits), _bf16_to_f32(V_bits))

    def set_current(self, layer, K_bits, V_bits):
        if layer not in self.nh:
            return
        self.current[layer] = (_bf16_to_f32(K_bits), _bf16_to_f32(V_bits))

    # ---- scoring and selection (Eq. 3) ----
    def roles(self, layer) -> FrameRoles:
        return frame_roles(self.nh[layer], self.S, self.W)

    def _seg(self, layer, t, j, head):
        lo, hi = segment_range(self.F, self.n, j)
        K = self.frames[layer][t][0]
        return K[lo:hi, head, :] if head is not None else np.transpose(K[lo:hi], (1, 0, 2))

    def _score_layer_head(self, layer, head):
        """(layer, head) whose keys score dynamic head `head` of layer `layer` (None = pooled)."""
        if self.source == "layer0_pooled":
            return 0, None
        return layer, head

    def _k_frame(self) -> int:
        return self.n if self.selection == "all" else keep_count(self.b, self.n)

    def scores(self, layer, head, exact: bool = False) -> dict:
        """Eq. 3 scores {t: [s_t^(0..n-1)]} over the scoreable frames; contract fp32 by
        default, fp64 definition with exact=True.  Under a comparison rule: the rule's
        ranking values instead."""
        sl, sh = self._score_layer_head(layer, head)
        out = {}
        if self.selection != "similarity":
            k = self._k_frame()
            for t in self.roles(sl).scoreable:
                out[t] = np.array([rule_value(self.selection, self.seed, t, j, self.n, k)
                                   for j in range(self.n)], dtype=np.float32)
            return out
        for t in self.roles(sl).scoreable:
            row = []
            for j in range(self.n):
                a, b = self._seg(sl, t, j, sh), self._seg(sl, t + 1, j, sh)
                row.append(cosine_fp64(a, b) if exact else segment_score_contract(a, b))
            out[t] = np.array(row, dtype=np.float64 if exact else np.float32)
        return out

    def kept(self, layer, head, exact: bool = False) -> list:
        """I_keep of Eq. 3 as ascending segment ids t*n + j (empty for a static head)."""
        if self.static[layer, head]:
            return []
        sc = self.scores(layer, head, exact=exact)
        if self.scope == "per_frame":
            k = self._k_frame()
            ids = []
            for t, row in sc.items():
                ids += [t * self.n + j for j in bottom_k(row, range(self.n), k)]
            return sorted(ids)
        cand_s, cand_i = [], []
        for t, row in sc.items():
            for j in range(self.n):
                cand_s.append(row[j])
                cand_i.append(t * self.n + j)
        n_keep = len(cand_i) if self.selection == "all" else keep_count(self.b, len(cand_i))
        return bottom_k(cand_s, cand_i, n_keep)

    # ---- Eq. 2 / Eq. 4 key sets and attention ----
    def current_frames(self, layer):
        nh = self.nh[layer]
        return range(nh, nh + self.C) if self.current[layer] is not None else range(0)

    def key_tokens(self, layer, head, kept=None) -> list:
        roles = self.roles(layer)
        cur = self.current_frames(layer)
        if self.static[layer, head]:
            return static_key_tokens(roles, self.F, cur, self.keep_anchor_static)
        if kept is None:
            kept = self.kept(layer, head)
        return dynamic_key_tokens(roles, self.F, self.n, kept, cur)

    def gather_kv(self, layer, head, kept=None):
        """K, V [Nk, D] fp64 of the head's key set."""
        F = self.F
        nh = self.nh[layer]
        ids = np.asarray(self.key_tokens(layer, head, kept), dtype=np.int64)
        Ks = np.empty((len(ids), self.D))
        Vs = np.empty((len(ids), self.D))
        frames = ids // F
        toks = ids % F
        for f in np.unique(frames):
            m = frames == f
            if f >= nh:
                Kc, Vc = self.current[layer]
                r = (f - nh) * F + toks[m]
                Ks[m], Vs[m] = Kc[r, head, :], Vc[r, head, :]
            else:
                Kf, Vf = self.frames[layer][int(f)]
                Ks[m], Vs[m] = Kf[toks[m], head, :], Vf[toks[m], head, :]
        return Ks, Vs

    def attend(self, layer, Q_bits, heads=None, rows=None, kept=None) -> np.ndarray:
        """O [rows, H, D] fp64: each head's queries over its Eq. 2 / Eq. 4 key set (Q K^T
        on e4m3 operands when the attention precision is "fp8_qk", both products when it is
        "fp8")."""
        Q = _bf16_to_f32(Q_bits)
        rows = np.arange(Q.shape[0]) if rows is None else np.asarray(rows)
        heads = range(self.H) if heads is None else heads
        O = np.full((len(rows), self.H, self.D), np.nan)
        for h in heads:
            K, V = self.gather_kv(layer, h, None if kept is None else kept.get(h))
            att = {"fp8_qk": attention_fp8_qk, "fp8": attention_fp8}.get(self.attn_precision,
                                                                         attention_fp64)
            O[:, h, :] = att(Q[rows, h, :], K, V)
        return O

    def view_length(self, layer, head) -> int:
        return len(self.key_tokens(layer, head))
