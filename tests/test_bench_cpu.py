"""Host-side logic of bench.py: replica aggregation over gloo ranks (world size 2, CPU) and the
CPU reference arm's output line.  No GPU needed."""
import json
import os
import subprocess
import sys
from pathlib import Path

import pytest
import torch
import torch.multiprocessing as mp

ROOT = Path(__file__).resolve().parent.parent


def _rank(rank, ws, port, out):
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=ws)
    sys.path.insert(0, str(ROOT))
    import bench
    # rank r processed (r + 1) * 1000 units in (r + 1) * 100 ms
    val, ms = bench.job_throughput(1000.0 * (rank + 1), 100.0 * (rank + 1), ws, device="cpu")
    out.put((rank, val, ms))
    dist.barrier()
    dist.destroy_process_group()


def test_replica_throughput_is_all_units_over_the_slowest_rank():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = 29517
    procs = [ctx.Process(target=_rank, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = [q.get(timeout=120) for _ in procs]
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for _, val, ms in res:
        assert ms == 200.0
        assert val == pytest.approx(3000.0 / 0.2)


def test_single_rank_needs_no_process_group():
    sys.path.insert(0, str(ROOT))
    import bench
    val, ms = bench.job_throughput(500.0, 250.0, 1)
    assert ms == 250.0 and val == pytest.approx(2000.0)


def test_reference_arm_prints_the_contract_line():
    env = dict(os.environ, CUDA_VISIBLE_DEVICES="")
    p = subprocess.run([sys.executable, str(ROOT / "bench.py"), "--impl", "reference", "--workload", "tiny",
                        "--steps", "1", "--warmup", "0"], capture_output=True, text=True, env=env, timeout=600)
    assert p.returncode == 0, p.stderr[-2000:]
    line = json.loads(p.stdout.strip().splitlines()[-1])
    assert line["impl"] == "reference" and line["metric"] == "retained prefill tokens/s"
    assert line["value"] > 0 and line["cpu_baseline"]["kind"] == "oracle" and line["cpu_baseline"]["cores"] >= 1
    assert line["e2e"]["h2d_bytes_per_step"] == 0 and line["e2e"]["value"] == line["value"]


def test_cpu_baseline_sample_is_clamped_to_a_small_workload():
    """The CPU-baseline sample asks for 8 tiles and 4 layers; the tiny scene has 4 tiles and a
    2-layer decoder, so the sample takes the whole scene and decoder instead of indexing past them."""
    sys.path.insert(0, str(ROOT))
    import bench
    from synth import workloads as W
    wl = W.TINY
    sc = W.make_scene(wl.scene, wl.decoder.vocab)
    t_tile, t_tok, cores, text = bench.oracle_sample(wl, sc, 8, 4, 10_000, torch.device("cpu"))
    assert t_tile > 0 and t_tok > 0 and cores >= 1
    assert "on 4 of 4 tiles" in text and "2 of 2 layers" in text
    assert f"one {wl.scene.S + wl.scene.n_v + wl.scene.Q}-token sequence" in text


def test_l2_note_and_traffic_belong_to_the_workload():
    """A workload whose inputs fit in L2 says it is flushed between steps, and the GEMM's DRAM
    traffic is reported only for the workload its ncu capture was taken on."""
    sys.path.insert(0, str(ROOT))
    import bench
    assert bench.l2_note(2 * 10**9, 13 * 10**9, False).startswith("inputs larger than L2")
    assert "flushed between timed steps" in bench.l2_note(2 * 10**6, 3 * 10**6, True)
    assert bench.gemm_traffic("tiny") is None
    t = bench.gemm_traffic(bench.PROFILED_WORKLOAD)
    assert t is None or t > 0


def test_select_gather_roofline_counts_the_algorithmic_bytes():
    from types import SimpleNamespace
    import bench
    sc = SimpleNamespace(S=35, Q=24, n_v=576, d=4096)
    n_kept, T = 3, 3 * (35 + 24) + 500  # 500 selected vision tokens
    r = bench.select_gather(n_kept, T, sc, 2, 0.01, 0.03, 6796.5)
    want = 3 * 576 * 4 + 2 * 500 * 4 + 500 * 4096 * 2 + 3 * 59 * 4096 * 2 + T * 4096 * 2
    assert r["bytes_per_query"] == want
    assert abs(r["ms_per_query"] - 0.04) < 1e-12
    assert abs(r["achieved_gbs"] - want / 0.04e-3 / 1e9) < 1e-6
    assert abs(r["frac"] - r["achieved_gbs"] / 6796.5) < 1e-12
    assert bench.select_gather(n_kept, T, sc, 2, 0.0, 0.0, 6796.5) is None
