"""Seeded streaming configurations of the GPU parity sweep (tests/test_parity_sweep_gpu.py);
tests/test_abi_cpu.py checks on the host that the library accepts every one of them."""
import numpy as np

import workloads as W

N_CASES = 48        # segments of 4-40 tokens: every attention row compared
N_LARGE = 16        # segments of 40-120 tokens: up to 2160 queries (sampled and boundary rows)


def sweep_case(i: int, large: bool = False) -> W.Workload:
    """Case i of the sweep (a pure function of i and the tier)."""
    rng = np.random.default_rng(7919 * (i + 1) + (104729 if large else 0))
    D = int(rng.choice([64, 128, 128]))
    precision = "bf16" if D == 64 else str(rng.choice(["bf16", "fp8_qk", "fp8"]))
    n = int(rng.choice([1, 2, 3, 4, 6]))
    seg = int(rng.integers(40, 121)) if large else int(rng.integers(4, 41))
    layers = int(rng.integers(1, 4))
    return W.ROLLING.with_(
        name=("sweep_large%02d" if large else "sweep%02d") % i, n_layers=layers,
        n_heads=int(rng.integers(1, 7)), head_dim=D,
        tokens_per_frame=n * seg, frames_per_chunk=int(rng.integers(1, 4)),
        n_sink_frames=int(rng.integers(0, 3)), window_frames=int(rng.choice([0, 2, 3, 4, 5, 7])),
        n_segments=n, keep_budget_permille=int(rng.integers(0, 1001)),
        select_scope=str(rng.choice(["per_frame", "pooled"])),
        score_source=str(rng.choice(["per_head", "layer0_pooled"])),
        incremental=bool(rng.integers(0, 2)), n_chunks=int(rng.integers(3, 7)),
        denoise_steps=int(rng.integers(1, 3)), rho_k=float(rng.uniform(0.6, 0.98)),
        scene_cut_every_chunks=int(rng.choice([0, 2, 3])), exact_half_static=False,
        static_fraction=float(rng.choice([0.0, 0.25, 0.5, 0.75, 1.0])), attn_precision=precision,
        seed=100 + i)
