"""Forcing-KV hot path on GB300: hybrid KV-cache compression (static structural pruning,
segment-similarity pruning) and chunk attention over the compressed cache.

Every step runs in the CUDA kernels of libfk.so behind the C ABI of include/fk.h; this
module only marshals arguments (torch tensors for device memory and streams).
"""
from __future__ import annotations

import ctypes

import numpy as np

from . import _lib as L
from ._lib import FkError, KERNEL_KINDS, STATUS_NAMES

__all__ = ["ForcingKVCache", "FkError", "KERNEL_KINDS", "STATUS_NAMES", "load_library",
           "head_profile", "classify_heads", "quantize_e4m3", "stream_read"]


def load_library():
    return L.load()


def _check(status: int, call: str) -> None:
    if status != L.FK_OK:
        raise FkError(status, call)


def _ptr(x) -> int:
    """Address of a bf16 tensor (torch, any device) or a uint16 numpy array of bf16 bits."""
    import torch
    if isinstance(x, torch.Tensor):
        if x.dtype != torch.bfloat16 or not x.is_contiguous():
            raise ValueError("expected a contiguous torch.bfloat16 tensor")
        return x.data_ptr()
    if isinstance(x, np.ndarray):
        if x.dtype != np.uint16 or not x.flags["C_CONTIGUOUS"]:
            raise ValueError("expected a C-contiguous uint16 array of bf16 bit patterns")
        return x.ctypes.data
    raise TypeError("unsupported tensor type %r" % type(x))


def _numel(x) -> int:
    return x.numel() if hasattr(x, "numel") and not isinstance(x, np.ndarray) else x.size


def _stream(stream) -> int | None:
    if stream is None:
        import torch
        if torch.cuda.is_available():
            return torch.cuda.current_stream().cuda_stream
        return None
    return getattr(stream, "cuda_stream", stream)


def head_profile(Q, K, n_generate: int, n_sink: int, n_transition: int, mass=None, status=None,
                 stream=None):
    """Offline head profiling (Sec. 4.1, Eq. 1) through fk_head_profile.

    Q [Nq, H, D] and K [Nk, H, D]: contiguous torch.bfloat16 CUDA tensors, keys ordered
    [generated | sink | other history | transition].  Adds each head's attention mass
    {A_Total, A_Generate, A_Transition, A_Sink} to `mass` (float64 [H, 4] on the device,
    created zeroed when None) and returns (mass, status); status is an int32 device tensor
    whose nonzero value means a bounded device wait expired."""
    import torch
    nq, H, D = Q.shape
    nk = K.shape[0]
    if tuple(K.shape[1:]) != (H, D):
        raise ValueError("Q and K disagree on heads / head_dim")
    if mass is None:
        mass = torch.zeros((H, 4), dtype=torch.float64, device=Q.device)
    if status is None:
        status = torch.zeros(1, dtype=torch.int32, device=Q.device)
    lib = L.load()
    _check(lib.fk_head_profile(_ptr(Q), _ptr(K), nq, nk, H, D, n_generate, n_sink, n_transition,
                               mass.data_ptr(), status.data_ptr(), _stream(stream)),
           "fk_head_profile")
    return mass, status


def quantize_e4m3(X, row_scaled: bool, q8=None, exps=None, stream=None):
    """E4M3 codes of a bf16 CUDA tensor [..., dim] as the FP8 attention path forms them
    (fk_quantize_e4m3): row_scaled=True scales each row by its power-of-two exponent (queries),
    False rounds unscaled (keys).  Returns (q8 uint8 tensor of X's shape, int8 exponents per
    row or None)."""
    import torch
    dim = X.shape[-1]
    rows = X.numel() // dim if dim else 0
    if q8 is None:
        q8 = torch.empty(X.shape, dtype=torch.uint8, device=X.device)
    if row_scaled and exps is None:
        exps = torch.empty(rows, dtype=torch.int8, device=X.device)
    lib = L.load()
    _check(lib.fk_quantize_e4m3(_ptr(X), rows, dim, 1 if row_scaled else 0, q8.data_ptr(),
                                exps.data_ptr() if exps is not None else None, _stream(stream)),
           "fk_quantize_e4m3")
    return q8, exps


def stream_read(X, nbytes: int | None = None, stream=None) -> None:
    """Read the first `nbytes` (default: all) of a CUDA tensor once (fk_stream_read): the
    event-timed floor of a launch that must read that many bytes."""
    if not X.is_contiguous():
        raise ValueError("expected a contiguous tensor")
    n = X.numel() * X.element_size() if nbytes is None else int(nbytes)
    if n > X.numel() * X.element_size():
        raise ValueError("nbytes exceeds the tensor")
    _check(L.load().fk_stream_read(X.data_ptr(), n, _stream(stream)), "fk_stream_read")


def classify_heads(mass, alpha: float = 0.8) -> np.ndarray:
    """Eq. 1 on masses [H, 4] (host copy): 1 = static, 0 = dynamic (fk_classify_heads)."""
    m = np.ascontiguousarray(np.asarray(mass, dtype=np.float64))
    H = m.shape[0]
    out = np.zeros(H, dtype=np.uint8)
    lib = L.load()
    _check(lib.fk_classify_heads(m.ctypes.data_as(ctypes.POINTER(ctypes.c_double)), H,
                                 int(round(alpha * 1000)),
                                 out.ctypes.data_as(ctypes.POINTER(ctypes.c_uint8))),
           "fk_classify_heads")
    return out


class ForcingKVCache:
    """One Forcing-KV cache (all layers of a model) on one GPU.

    Tensors are bf16 [tokens, n_heads, head_dim]; device or host memory.  Calls are
    asynchronous on `stream` (default: torch's current stream)."""

    def __init__(self, *, n_layers, n_heads, head_dim, tokens_per_frame, frames_per_chunk,
                 n_sink_frames, window_frames, n_segments, keep_budget_permille,
                 head_is_static, select_scope="per_frame", score_source="per_head",
                 incremental=False, max_history_frames=64, device=0, selection="similarity",
                 select_seed=0, static_drop_anchor=False, attn_precision="bf16"):
        self._lib = L.load()
        self._h = ctypes.c_void_p()
        hm = np.ascontiguousarray(np.asarray(head_is_static, dtype=np.uint8).reshape(-1))
        if hm.size != n_layers * n_heads:
            raise ValueError("head_is_static must have n_layers * n_heads entries")
        self._map = hm
        self.cfg = L.FkConfig(
            n_layers, n_heads, head_dim, tokens_per_frame, frames_per_chunk, n_sink_frames,
            window_frames, n_segments, keep_budget_permille,
            {"per_frame": L.FK_SCOPE_PER_FRAME, "pooled": L.FK_SCOPE_POOLED}[select_scope],
            {"per_head": L.FK_SCORE_PER_HEAD, "layer0_pooled": L.FK_SCORE_LAYER0_POOLED}[score_source],
            1 if incremental else 0, max_history_frames, device,
            hm.ctypes.data_as(ctypes.POINTER(ctypes.c_uint8)),
            L.FK_SELECT[selection], select_seed & 0xFFFFFFFF, 1 if static_drop_anchor else 0,
            L.FK_ATTN[attn_precision])
        self.n_layers, self.n_heads, self.head_dim = n_layers, n_heads, head_dim
        self.F, self.C, self.n_segments = tokens_per_frame, frames_per_chunk, n_segments
        self.device = device
        _check(self._lib.fk_create(ctypes.byref(self.cfg), ctypes.byref(self._h)), "fk_create")

    @classmethod
    def from_workload(cls, w, head_is_static, device=0, **over):
        kw = dict(n_layers=w.n_layers, n_heads=w.n_heads, head_dim=w.head_dim,
                  tokens_per_frame=w.tokens_per_frame, frames_per_chunk=w.frames_per_chunk,
                  n_sink_frames=w.n_sink_frames, window_frames=w.window_frames,
                  n_segments=w.n_segments, keep_budget_permille=w.keep_budget_permille,
                  head_is_static=head_is_static, select_scope=w.select_scope,
                  score_source=w.score_source, incremental=w.incremental,
                  max_history_frames=max(1, w.max_history_frames()), device=device,
                  selection=w.selection, select_seed=w.select_seed,
                  static_drop_anchor=w.static_drop_anchor, attn_precision=w.attn_precision)
        kw.update(over)
        return cls(**kw)

    # ---- lifetime
    def close(self):
        if getattr(self, "_h", None) and self._h.value:
            self._lib.fk_destroy(self._h)
            self._h = ctypes.c_void_p()

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def __enter__(self):
        return self

    def __exit__(self, *exc):
        self.close()

    # ---- cache updates
    def append_frames(self, layer, K, V, stream=None):
        nf = _numel(K) // (self.F * self.n_heads * self.head_dim)
        _check(self._lib.fk_append_frames(self._h, layer, _ptr(K), _ptr(V), nf, _stream(stream)),
               "fk_append_frames")

    def append_chunk(self, layer, K, V, stream=None):
        _check(self._lib.fk_append_chunk(self._h, layer, _ptr(K), _ptr(V), _stream(stream)),
               "fk_append_chunk")

    def set_current(self, layer, K, V, stream=None):
        _check(self._lib.fk_set_current(self._h, layer, _ptr(K), _ptr(V), _stream(stream)),
               "fk_set_current")

    def compress(self, stream=None):
        _check(self._lib.fk_compress(self._h, _stream(stream)), "fk_compress")

    def attend(self, layer, Q, O=None, stream=None):
        if O is None:
            import torch
            O = torch.empty_like(Q)
        _check(self._lib.fk_attend(self._h, layer, _ptr(Q), _ptr(O), _stream(stream)), "fk_attend")
        return O

    # ---- inspection
    def kept(self, layer, head, stream=None) -> list:
        n = ctypes.c_int(0)
        st = self._lib.fk_get_kept(self._h, layer, head, None, 0, ctypes.byref(n), _stream(stream))
        if n.value == 0:
            _check(st, "fk_get_kept")
            return []
        buf = (ctypes.c_int32 * n.value)()
        _check(self._lib.fk_get_kept(self._h, layer, head, buf, n.value, ctypes.byref(n),
                                     _stream(stream)), "fk_get_kept")
        return list(buf)

    def scores(self, layer, head, stream=None):
        """(first_frame, fp32 array [n_frames, n_segments]) of the scoreable frames."""
        first, nfr = ctypes.c_int(0), ctypes.c_int(0)
        cap = 1 << 16
        buf = np.zeros(cap, dtype=np.float32)
        _check(self._lib.fk_get_scores(self._h, layer, head,
                                       buf.ctypes.data_as(ctypes.POINTER(ctypes.c_float)), cap,
                                       ctypes.byref(first), ctypes.byref(nfr), _stream(stream)),
               "fk_get_scores")
        return first.value, buf[: nfr.value * self.n_segments].reshape(nfr.value, self.n_segments).copy()

    def key_count(self, layer, head) -> int:
        n = ctypes.c_int(0)
        _check(self._lib.fk_key_count(self._h, layer, head, ctypes.byref(n)), "fk_key_count")
        return n.value

    def cache_bytes(self) -> int:
        return int(self._lib.fk_cache_bytes(self._h))

    def reserved_bytes(self) -> int:
        return int(self._lib.fk_reserved_bytes(self._h))

    def sync_status(self, stream=None) -> int:
        """Synchronize and return the device status (FK_OK, FK_ERR_RANGE, FK_ERR_TIMEOUT)."""
        return int(self._lib.fk_sync_status(self._h, _stream(stream)))

    # ---- timing
    def profile_enable(self, on=True):
        _check(self._lib.fk_profile_enable(self._h, 1 if on else 0), "fk_profile_enable")

    def profile_reset(self):
        _check(self._lib.fk_profile_reset(self._h), "fk_profile_reset")

    def profile_read(self, kind: str):
        ms, n = ctypes.c_double(0), ctypes.c_int64(0)
        _check(self._lib.fk_profile_read(self._h, KERNEL_KINDS[kind], ctypes.byref(ms),
                                         ctypes.byref(n)), "fk_profile_read")
        return ms.value, n.value

    def wait_selftest(self, limit_us: int = 20000, stream=None) -> None:
        """Run the bounded-wait self-test (fk_wait_selftest): the next sync_status() reports
        FK_ERR_TIMEOUT."""
        _check(self._lib.fk_wait_selftest(self._h, int(limit_us), _stream(stream)), "fk_wait_selftest")

    def set_host_overlap(self, on: bool = True) -> None:
        """Overlap host transfers with queued work (see fk_set_host_overlap): host inputs must
        be final at call time; host outputs are complete after wait_outputs() (or
        sync_status()) and a synchronization of the stream."""
        _check(self._lib.fk_set_host_overlap(self._h, 1 if on else 0), "fk_set_host_overlap")

    def wait_outputs(self, stream=None) -> None:
        """Make the stream wait for pending host-output copies (fk_wait_outputs)."""
        _check(self._lib.fk_wait_outputs(self._h, _stream(stream)), "fk_wait_outputs")

    def launch_count(self) -> int:
        return int(self._lib.fk_launch_count(self._h))
