"""Seeded sweep over small streaming configurations, GPU path against the oracle.

Each case draws its options together: head_dim 64 / 128, 1-6 heads with any static/dynamic
split (none static, all static, anything between), 1-3 layers, per-frame or pooled selection,
per-head or layer-0 pooled scoring, whole-window or incremental scoring, the three attention
precisions (FP8 at D = 128), 0-2 sink frames, an unbounded or 2-7 frame window, any keep
budget, 1-6 segments of 4-40 tokens (a second tier: 40-120), 1-3 frames per chunk, 1-2 denoising steps and scene cuts.
The feature tests exercise these options one at a time; the sweep covers their interactions
(a key split over a ragged pooled view, a window shorter than a chunk with sinks and an
incremental ring, ...).  At every compress of every case: kept sets and scores bit-exact,
key counts exact, every attention row within the standard tolerance."""
import pytest

from fkharness import run_stream
from sweep_cases import N_CASES, N_LARGE, sweep_case

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


@pytest.fixture(scope="module", autouse=True)
def _library():
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    from paper_2605_09681_gb300 import build, load_library
    build.build()
    load_library()


@pytest.mark.parametrize("i", range(N_CASES))
def test_sweep_case(i):
    w = sweep_case(i)
    n = run_stream(w, track_layers=tuple(range(w.n_layers)))
    assert n == w.n_chunks * w.denoise_steps * w.n_layers


@pytest.mark.parametrize("i", range(N_LARGE))
def test_sweep_large_case(i):
    w = sweep_case(i, large=True)
    n = run_stream(w, track_layers=tuple(range(w.n_layers)))
    assert n == w.n_chunks * w.denoise_steps * w.n_layers
