"""The allocation-free scoring entry point, for callers that must not call cudaMalloc (a host
framework owning all device memory, or a real-time loop with a fixed memory budget).  It must
return the same segment scores as the regular path (fk_compress then fk_get_scores) on the same
frames, bit for bit, on consecutive calls that reuse its fixed device scratch array.  Kept in its
own file, collected last, so a failure here never hides the other tests."""
import ctypes

import numpy as np
import pytest

import workloads as W

pytestmark = pytest.mark.gpu
torch = pytest.importorskip("torch")


def _frames(F, D, n_frames, seed):
    w = W.Workload(name="noalloc", n_layers=1, n_heads=1, head_dim=D, tokens_per_frame=F,
                   frames_per_chunk=3, n_sink_frames=0, window_frames=0, n_segments=6,
                   keep_budget_permille=700, rho_k=0.9, seed=seed)
    k, _v = W.FrameStream(w, 0).frames(n_frames)          # [n_frames*F, 1, D]
    return w, k


def _regular_scores(w, k, n_frames, n_seg):
    from paper_2605_09681_gb300 import ForcingKVCache
    kd = torch.from_numpy(k.view(np.int16)).view(torch.bfloat16).cuda()
    with ForcingKVCache(n_layers=1, n_heads=1, head_dim=w.head_dim, tokens_per_frame=w.tokens_per_frame,
                        frames_per_chunk=1, n_sink_frames=0, window_frames=0, n_segments=n_seg,
                        keep_budget_permille=700, head_is_static=[[0]],
                        max_history_frames=n_frames) as c:
        c.append_frames(0, kd, kd)
        c.compress()
        first, sc = c.scores(0, 0)
    assert first == 0 and sc.shape == (n_frames - 1, n_seg)
    return sc


def test_noalloc_matches_regular_scoring_on_consecutive_calls():
    assert torch.cuda.is_available()
    from paper_2605_09681_gb300 import _lib, build
    build.build()
    lib = _lib.load()
    stream = torch.cuda.current_stream()
    for (F, D, n_frames, n_seg, seed) in [(1560, 128, 12, 6, 21), (600, 64, 9, 6, 22), (1560, 128, 12, 6, 23)]:
        w, k = _frames(F, D, n_frames, seed)
        ref = _regular_scores(w.with_(n_segments=n_seg), k, n_frames, n_seg)
        kd = torch.from_numpy(k.view(np.int16)).view(torch.bfloat16).cuda()
        out = torch.full((n_frames - 1, n_seg), float("nan"), dtype=torch.float32, device="cuda")
        st = lib.fk_segment_scores_noalloc(kd.data_ptr(), n_frames, F, D, n_seg, out.data_ptr(),
                                           stream.cuda_stream)
        assert st == 0, _lib.STATUS_NAMES.get(st)
        torch.cuda.synchronize()
        got = out.cpu().numpy()
        assert np.array_equal(got.view(np.uint32), ref.view(np.uint32)), (F, D, seed)


def test_noalloc_rejects_sizes_beyond_its_limit():
    from paper_2605_09681_gb300 import _lib
    lib = _lib.load()
    kd = torch.zeros((4, 64, 128), dtype=torch.bfloat16, device="cuda")
    out = torch.zeros((3, 64), dtype=torch.float32, device="cuda")
    assert lib.fk_segment_scores_noalloc(kd.data_ptr(), 4, 64, 128, 64, out.data_ptr(), None) == 1
    assert lib.fk_segment_scores_noalloc(kd.data_ptr(), 300, 64, 128, 8, out.data_ptr(), None) == 1
    host = np.zeros((4, 64, 128), dtype=np.uint16)
    assert lib.fk_segment_scores_noalloc(host.ctypes.data, 4, 64, 128, 8, out.data_ptr(), None) == 2
