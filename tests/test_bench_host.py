"""Host logic of bench.py that needs no GPU: the sweep definition, whole-job
aggregation, the max-over-ranks reduction on two gloo ranks, the reference
arm's rank handling and its JSON line, and the oracle's row sample of the
sweep operands."""
import json
import os
import socket
import subprocess
import sys

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)
import bench  # noqa: E402
from paper_1810_09958_gb300 import synth  # noqa: E402


def test_sweep_has_32_problems_with_both_layouts():
    probs = bench.sweep_problems()
    assert len(probs) == 32
    assert {tA for *_, tA in probs} == {0, 1}
    assert {(M, K) for M, N, K, tA in probs} == set(bench.SWEEP_MK)
    assert {N for M, N, K, tA in probs} == set(bench.SWEEP_N)


def test_gemm_work_formulas():
    assert bench.gemm_flops(2, 3, 4) == 48
    assert bench.gemm_bytes(2, 3, 4) == 2 * 2 * 4 + 2 * 4 * 3 + 4 * 2 * 3
    assert bench.gemm_bytes(2, 3, 4, beta=True) == 2 * 2 * 4 + 2 * 4 * 3 + 8 * 2 * 3


def test_whole_job_value_is_weak_scaling_aggregate():
    # 2 ranks, each 1 TFLOP per step, 10 steps, slowest rank 10 ms -> 2000 TFLOP/s.
    assert bench.whole_job_tflops(1e12, 10, 2, 10.0) == pytest.approx(2000.0)


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _rank_main(rank, world, port, out_q):
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        bench.barrier()
        got = bench.reduce_max(float(rank + 1) * 1.5)
        out_q.put((rank, got))
    finally:
        dist.destroy_process_group()


def test_reduce_max_over_two_gloo_ranks():
    import torch.multiprocessing as mp
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=120)
        assert p.exitcode == 0
    res = dict(q.get(timeout=10) for _ in range(2))
    assert res == {0: 3.0, 1: 3.0}


def test_reduce_max_without_process_group_is_identity():
    assert bench.reduce_max(4.25) == 4.25


def test_reference_arm_other_ranks_exit_silently():
    env = dict(os.environ, RANK="1", WORLD_SIZE="2", LOCAL_RANK="1")
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference",
                        "--steps", "1", "--warmup", "3"], env=env, capture_output=True, text=True,
                       timeout=120)
    assert r.returncode == 0
    assert r.stdout.strip() == ""


def test_reference_arm_prints_the_contract_line():
    """Rank 0 of the reference arm (the fp64 oracle on the host cores) prints
    one JSON line with the contract's keys; its end-to-end figure is its own
    value with no host-device copies."""
    env = {k: v for k, v in os.environ.items() if k not in ("RANK", "WORLD_SIZE", "LOCAL_RANK")}
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference",
                        "--steps", "1", "--warmup", "3"], env=env, capture_output=True, text=True,
                       timeout=600)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [l for l in r.stdout.splitlines() if l.strip()]
    assert len(lines) == 1
    d = json.loads(lines[0])
    for key in ("metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step", "higher_is_better",
                "scaling", "vs_baseline", "dtype", "data", "config"):
        assert key in d, key
    assert d["impl"] == "reference" and d["warmup"] >= 3 and d["steps"] == 1
    assert d["value"] > 0 and d["unit"] == "TFLOP/s" and d["higher_is_better"] is True
    cb = d["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["cores"] >= 1 and cb["sample"] and cb["value"] == d["value"]
    assert d["e2e"] == {"value": d["value"], "unit": d["unit"], "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}
    assert "workload" in d["config"]


def test_oracle_row_sample_draws_the_same_rows():
    """The CPU baseline's sampled rows of op(A) are exactly those rows of the
    operands the GPU arm generates (same counter-based streams)."""
    stride = 97
    ops = bench.sample_operands(stride)
    for (M, N, K, tA), (R, N2, K2, A_sub, B) in zip(bench.sweep_problems(), ops):
        if (M, K) != (1760, 1760) or N != 16:
            continue
        seed = synth.stream_seed(synth.BASE_SEED, 1, M, K, N, tA)
        A_full = synth.bf16_uniform(synth.stream_seed(seed, 1), (K, M) if tA else (M, K))
        opA = A_full.T if tA else A_full
        rows = bench.row_sample(M, stride)
        assert R == rows.size and N2 == N and K2 == K
        assert np.array_equal(A_sub, opA[rows])
        assert np.array_equal(B, synth.bf16_uniform(synth.stream_seed(seed, 2), (K, N)))
