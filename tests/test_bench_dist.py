"""The multi-process host logic of bench.py (replicas on N GPUs): barrier and the maximum of the
ranks' timings, run as two gloo ranks on the CPU."""
import os
import socket

import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _rank(rank, world, port, results):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), WORLD_SIZE=str(world),
                      RANK=str(rank), LOCAL_RANK=str(rank))
    import bench
    r, w, lr = bench._dist()
    assert (r, w, lr) == (rank, world, rank)
    bench.barrier(w)
    results[rank] = bench.reduce_max(10.0 + 5.0 * rank, w)
    bench.barrier(w)
    import torch.distributed as dist
    dist.destroy_process_group()


def test_two_rank_timing_reduction():
    ctx = mp.get_context("spawn")
    manager = ctx.Manager()
    results = manager.dict()
    port = _free_port()
    procs = [ctx.Process(target=_rank, args=(r, 2, port, results)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=120)
        assert p.exitcode == 0
    assert dict(results) == {0: 15.0, 1: 15.0}


def test_single_rank_needs_no_process_group():
    import bench
    assert bench.reduce_max(3.5, 1) == 3.5
    bench.barrier(1)


def test_reference_arm_json_contract():
    # the oracle arm on the host cores: one JSON line with the base contract's keys, the
    # reference markers, and the same workload config as the GPU arm
    import json
    import subprocess
    import sys
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference",
                        "--steps", "1", "--warmup", "3"], capture_output=True, text=True,
                       timeout=600, cwd=ROOT)
    assert r.returncode == 0, r.stderr[-2000:]
    line = json.loads(r.stdout.strip().splitlines()[-1])
    for k in ("metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step",
              "higher_is_better", "scaling", "vs_baseline", "dtype", "data", "config", "e2e"):
        assert k in line, k
    assert line["impl"] == "reference" and line["value"] > 0 and line["higher_is_better"] is True
    assert (line["steps"], line["warmup"], line["n_gpus"]) == (1, 3, 1)
    cb = line["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["cores"] >= 1 and cb["sample"] and cb["value"] == line["value"]
    assert line["e2e"] == {"value": line["value"], "unit": line["unit"], "h2d_bytes_per_step": 0,
                           "d2h_bytes_per_step": 0}
    cfg = line["config"]
    assert cfg["keys_per_head"] == [7800, 7800, 25480, 25480, 25480, 7800, 7800, 25480, 7800,
                                    25480, 7800, 25480]
    assert cfg["queries"] == 4680 and cfg["head_dim"] == 128 and cfg["heads"] == 12
    assert line["extrapolated"] is True and line["measured_ms_per_step"] > 0


def test_algorithmic_work_of_the_480p_step():
    # the figures every roofline fraction divides by, worked out by hand for the 480P layer:
    # 6 static heads see 7800 keys (current 4680 + sink 1560 + anchor 1560), 6 dynamic heads
    # 25480 (current + sink + anchor + 17 frames x 4 kept segments x 260 tokens)
    import bench
    w = bench._workload("480p_layer")
    keys = [7800] * 6 + [25480] * 6
    alg = bench._algorithmic(w, keys)
    assert alg["attn_flops"] == 4 * 4680 * 128 * (6 * 7800 + 6 * 25480)            # 478.47 GFLOP
    # the scoring kernel reads frames 1..15 (the frame before the retired chunk included); the
    # current-chunk kernel forms the sums of the retired frames 16..18 as it moves them
    assert alg["score_fused"] and alg["score_bytes"] == 6 * 15 * 1560 * 128 * 2    # 35.94 MB
    # chunk K, V read + written; each static head's anchor slot and each dynamic head's three
    # retired frames (K, V read + written); each dynamic head's partner key frame; each dynamic
    # head's new anchor frame (K, V) written into its view
    assert alg["append_bytes"] == (2 * 2 * 4680 * 12 * 128 * 2 + 6 * 2 * 2 * 1560 * 128 * 2
                                   + 6 * 2 * 2 * 3 * 1560 * 128 * 2 + 6 * 1560 * 128 * 2
                                   + 6 * 2 * 1560 * 128 * 2)
    assert alg["compact_bytes"] == 6 * 17 * 4 * 260 * 128 * 2 * 2 * 2             # 108.7 MB
    cfg = bench._config(w, keys)
    assert cfg["queries"] == 4680 and cfg["history_frames"] == 18 and cfg["keys_per_head"] == keys


def test_both_arms_print_the_same_config():
    # the reference arm's config is built by the same function from the same workload and key
    # counts, and carries no arm-specific field
    import bench
    import workloads as W
    w = bench._workload("480p_layer")
    keys = [7800 if s else 25480 for s in W.head_map(w)[0]]
    assert bench._config(w, keys) == bench._config(bench._workload("480p_layer"), list(keys))
