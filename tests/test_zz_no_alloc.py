"""The allocation-free scoring entry point, for callers that must not call cudaMalloc (a host
framework owning all device memory, or a real-time loop with a fixed memory budget).  It must
return the same segment scores as the regular path (fk_compress then fk_get_scores) on the same
frames, bit for bit, on consecutive calls that reuse its fixed device scratch array, including
calls at its documented limits and calls of different sizes back to back on one stream.  Kept
in its own file, collected last, so a failure here never hides the other tests."""
import numpy as np
import pytest

import workloads as W

pytestmark = pytest.mark.gpu
torch = pytest.importorskip("torch")


def _frames(F, D, n_frames, seed):
    w = W.Workload(name="noalloc", n_layers=1, n_heads=1, head_dim=D, tokens_per_frame=F,
                   frames_per_chunk=3, n_sink_frames=0, window_frames=0, n_segments=1,
                   keep_budget_permille=700, rho_k=0.9, seed=seed)
    k, _v = W.FrameStream(w, 0).frames(n_frames)          # [n_frames*F, 1, D]
    return k


def _dev(k):
    return torch.from_numpy(np.ascontiguousarray(k).view(np.int16)).view(torch.bfloat16).cuda()


def _regular_scores(k, F, D, n_frames, n_seg):
    from paper_2605_09681_gb300 import ForcingKVCache
    kd = _dev(k)
    with ForcingKVCache(n_layers=1, n_heads=1, head_dim=D, tokens_per_frame=F,
                        frames_per_chunk=1, n_sink_frames=0, window_frames=0, n_segments=n_seg,
                        keep_budget_permille=700, head_is_static=[[0]],
                        max_history_frames=n_frames) as c:
        c.append_frames(0, kd, kd)
        c.compress()
        first, sc = c.scores(0, 0)
        assert c.sync_status() == 0
    assert first == 0 and sc.shape == (n_frames - 1, n_seg)
    return sc


@pytest.fixture(scope="module")
def lib():
    assert torch.cuda.is_available()
    from paper_2605_09681_gb300 import _lib, build
    build.build()
    return _lib.load()


# (tokens_per_frame, head_dim, n_frames, n_segments, seed): a 480P-sized frame, small frames,
# and both documented limits (256 frames; 32 segments; frames x segments = 4096)
CASES = [(1560, 128, 12, 6, 21), (600, 64, 9, 6, 22), (1560, 128, 12, 6, 23),
         (64, 64, 256, 16, 24), (64, 128, 128, 32, 25), (96, 128, 2, 32, 26), (64, 64, 256, 16, 27)]


def test_noalloc_matches_regular_scoring_on_consecutive_calls(lib):
    from paper_2605_09681_gb300 import _lib
    stream = torch.cuda.current_stream()
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    refs, outs, keep = [], [], []
    for (F, D, n_frames, n_seg, seed) in CASES:
        k = _frames(F, D, n_frames, seed)
        refs.append(_regular_scores(k, F, D, n_frames, n_seg))
        keep.append(_dev(k))
    torch.cuda.synchronize()
    # every call queued back to back on one stream, sizes changing from call to call
    for (F, D, n_frames, n_seg, _seed), kd in zip(CASES, keep):
        out = torch.full((n_frames - 1, n_seg), float("nan"), dtype=torch.float32, device="cuda")
        st = lib.fk_segment_scores_noalloc(kd.data_ptr(), n_frames, F, D, n_seg, out.data_ptr(),
                                           status.data_ptr(), stream.cuda_stream)
        assert st == 0, _lib.STATUS_NAMES.get(st)
        outs.append(out)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    for case, ref, out in zip(CASES, refs, outs):
        got = out.cpu().numpy()
        assert np.array_equal(got.view(np.uint32), ref.view(np.uint32)), case
    # the same calls again without the status word (conditions then go unreported)
    for (F, D, n_frames, n_seg, _seed), kd, ref in zip(CASES[:2], keep, refs):
        out = torch.zeros((n_frames - 1, n_seg), dtype=torch.float32, device="cuda")
        assert lib.fk_segment_scores_noalloc(kd.data_ptr(), n_frames, F, D, n_seg, out.data_ptr(),
                                             None, stream.cuda_stream) == 0
        torch.cuda.synchronize()
        assert np.array_equal(out.cpu().numpy().view(np.uint32), ref.view(np.uint32))


def test_noalloc_reports_the_scoring_precondition(lib):
    # one token whose squared key norm is above 2^23 sets bit 1 of the caller's status word
    F, D, n_frames, n_seg = 64, 64, 4, 8
    k = W.bf16_bits_to_f32(_frames(F, D, n_frames, 31)).copy()
    k[F + 5] = 400.0                                      # 64 x 400^2 > 2^23
    kd = _dev(W.to_bf16_bits(k))
    out = torch.zeros((n_frames - 1, n_seg), dtype=torch.float32, device="cuda")
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    assert lib.fk_segment_scores_noalloc(kd.data_ptr(), n_frames, F, D, n_seg, out.data_ptr(),
                                         status.data_ptr(), None) == 0
    torch.cuda.synchronize()
    assert int(status.item()) & 1
    # a clean call afterwards leaves a fresh status word at zero
    status.zero_()
    kd = _dev(_frames(F, D, n_frames, 32))
    assert lib.fk_segment_scores_noalloc(kd.data_ptr(), n_frames, F, D, n_seg, out.data_ptr(),
                                         status.data_ptr(), None) == 0
    torch.cuda.synchronize()
    assert int(status.item()) == 0


def test_noalloc_rejects_sizes_beyond_its_limit(lib):
    kd = torch.zeros((4, 64, 128), dtype=torch.bfloat16, device="cuda")
    out = torch.zeros((3, 64), dtype=torch.float32, device="cuda")
    f = lib.fk_segment_scores_noalloc
    assert f(kd.data_ptr(), 4, 64, 128, 64, out.data_ptr(), None, None) == 1     # 64 segments
    assert f(kd.data_ptr(), 300, 64, 128, 8, out.data_ptr(), None, None) == 1    # 300 frames
    assert f(kd.data_ptr(), 256, 64, 128, 32, out.data_ptr(), None, None) == 1   # 8192 cells
    host = np.zeros((4, 64, 128), dtype=np.uint16)
    assert f(host.ctypes.data, 4, 64, 128, 8, out.data_ptr(), None, None) == 2   # host K
    hs = np.zeros(1, dtype=np.int32)
    assert f(kd.data_ptr(), 4, 64, 128, 8, out.data_ptr(), hs.ctypes.data, None) == 2   # host status
