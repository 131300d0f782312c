"""Benchmark of Rift's hot path on GB300: one step = one scene query through every stage
(query prep, Eq. 1 scoring, kNN smoothing, min-max + tau pruning, Eq. 2 budgets, top-b
selection, ragged packing, 32-layer prefill of the retained sequences).

    python bench.py [--gpus N] [--steps K] [--warmup W] [--workload rift400_7b] [--impl reference]

Prints one JSON line.  value = retained prefill tokens/s over all ranks (each rank runs its
own replica of the scene query: the queries are independent, there is no collective on the
data path).  Inputs (X: 1.9 GB, weights: 13 GB) are larger than L2, so no flush is needed.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import threading
import time
from pathlib import Path

ROOT = Path(__file__).resolve().parent
sys.path.insert(0, str(ROOT))

import torch  # noqa: E402

from synth import rng, workloads as W  # noqa: E402

METRIC = "retained prefill tokens/s"
UNIT = "tokens/s"


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=10)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--workload", default="rift400_7b", choices=sorted(W.WORKLOADS))
    ap.add_argument("--impl", default="rift", choices=["rift", "reference"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--e2e-steps", type=int, default=20)
    ap.add_argument("--no-decode", action="store_true", help="skip the decode-step measurement")
    ap.add_argument("--no-shared-prefix", action="store_true", help="skip the shared-prefix measurement")
    ap.add_argument("--no-batch", action="store_true", help="skip the multi-query batch measurement")
    ap.add_argument("--ncu-summary", metavar="CSV", help="summarise an ncu launch list (gpu__time_duration.sum) and exit")
    ap.add_argument("--sweep", action="store_true",
                    help="scoring/select/gather-only sweep over N in {100, 400, 1600, 6400} tiles (one JSON line per N)")
    ap.add_argument("--kernel-case", choices=["prefill", "prefill_full", "score", "decode", "merge", "attention"],
                    help="small profiling case: 'prefill' = one 7B-shaped layer over 12 sequences (T = 4092), "
                         "'prefill_full' = one 7B-shaped layer over the 400-tile query's retained length mix "
                         "(73 sequences, T = 23,819), 'score' = Eq. 1 scoring of 64 tiles (302 MB of tokens), "
                         "'attention' = the varlen attention alone over ~23.6K rows of sequences of one length, "
                         "for lengths 131 to 4096 (CUDA events, one JSON line per length); the others run 3 times")
    return ap.parse_args()


def ncu_summary(path: str) -> str:
    """Per kernel of an ncu --csv launch list: launches, total device time, share and, when the
    list has dram__bytes_read.sum / dram__bytes_write.sum, DRAM traffic.  Ends with the GEMM
    traffic block that bench.py reads back (mean DRAM bytes per gemm_tc_kernel launch and the
    hash of the gemm_tc.cu it was measured on)."""
    import csv
    import hashlib
    with open(path) as f:
        rows = list(csv.DictReader([ln for ln in f if ln.startswith('"')]))
    tscale = {"ns": 1e-6, "nsecond": 1e-6, "us": 1e-3, "usecond": 1e-3, "ms": 1.0, "msecond": 1.0}
    bscale = {"byte": 1.0, "Kbyte": 1e3, "Mbyte": 1e6, "Gbyte": 1e9, "Tbyte": 1e12}
    launches = {}
    for r in rows:
        d = launches.setdefault(r["ID"], {"name": r["Kernel Name"].split("(")[0]})
        v = float(r["Metric Value"].replace(",", ""))
        if r["Metric Name"] == "gpu__time_duration.sum":
            d["ms"] = v * tscale.get(r["Metric Unit"], 1e-6)
        elif r["Metric Name"] in ("dram__bytes_read.sum", "dram__bytes_write.sum"):
            d[r["Metric Name"]] = v * bscale.get(r["Metric Unit"], 1.0)
    agg = {}
    for d in launches.values():
        a = agg.setdefault(d["name"], [0, 0.0, 0.0, 0.0])
        a[0] += 1
        a[1] += d.get("ms", 0.0)
        a[2] += d.get("dram__bytes_read.sum", 0.0)
        a[3] += d.get("dram__bytes_write.sum", 0.0)
    total = sum(v[1] for v in agg.values())
    dram = any(v[2] or v[3] for v in agg.values())
    out = [f"{'kernel':<46} {'launches':>8} {'total ms':>10} {'share':>7}" + (
        f" {'DRAM rd GB':>10} {'DRAM wr GB':>10} {'GB/s':>6}" if dram else "")]
    for name, (n, t, rd, wr) in sorted(agg.items(), key=lambda kv: -kv[1][1]):
        line = f"{name[:46]:<46} {n:>8} {t:>10.3f} {100 * t / total:>6.2f}%"
        if dram:
            line += f" {rd / 1e9:>10.3f} {wr / 1e9:>10.3f} {(rd + wr) / 1e6 / t if t else 0:>6.0f}"
        out.append(line)
    out.append(f"{'all':<46} {sum(v[0] for v in agg.values()):>8} {total:>10.3f}")
    gemm = [(n, a) for n, a in agg.items() if "gemm_tc_kernel" in n]
    if dram and gemm:
        n = sum(a[0] for _, a in gemm)
        b = sum(a[2] + a[3] for _, a in gemm)
        src = ROOT / "paper_2609_29029_gb300" / "csrc" / "gemm_tc.cu"
        out += ["", "GEMM traffic used by bench.py (mean over the gemm_tc_kernel launches of the list):", "",
                "- kernel: gemm_tc_kernel",
                f"- source_sha256_16: {hashlib.sha256(src.read_bytes()).hexdigest()[:16]}",
                f"- dram_bytes_per_launch: {int(b / n)}", f"- launches: {n}"]
    return "\n".join(out)


# ------------------------------------------------------------------------------------------ dist

def dist_setup():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if ws > 1:
        import torch.distributed as dist
        torch.cuda.set_device(local)
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    return ws, rank, local


def barrier(ws):
    if ws > 1:
        import torch.distributed as dist
        dist.barrier()


def _reduce(x: float, ws: int, op: str, device) -> float:
    if ws == 1:
        return x
    import torch.distributed as dist
    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX if op == "max" else dist.ReduceOp.SUM)
    return float(t.item())


def reduce_max(x: float, ws: int, device="cuda") -> float:
    return _reduce(x, ws, "max", device)


def reduce_sum(x: float, ws: int, device="cuda") -> float:
    return _reduce(x, ws, "sum", device)


def job_throughput(units_this_rank: float, ms_this_rank: float, ws: int, device="cuda"):
    """Whole-job rate over replicas: units of all ranks / the slowest rank's time."""
    ms_max = reduce_max(ms_this_rank, ws, device)
    units = reduce_sum(units_this_rank, ws, device)
    return units / (ms_max / 1e3), ms_max


# ------------------------------------------------------------------------------------------ clocks

class ClockSampler:
    """nvidia-smi samples of SM clock and throttle reasons while the timed region runs."""

    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.hw_slowdown,"
              "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
              "clocks_event_reasons.sw_power_cap")

    def __init__(self, device_index: int):
        self.idx = device_index
        self.proc = None
        self.lines = []

    def __enter__(self):
        try:
            uuid = "GPU-" + str(torch.cuda.get_device_properties(self.idx).uuid)
            self.proc = subprocess.Popen(["nvidia-smi", "-i", uuid, f"--query-gpu={self.FIELDS}",
                                          "--format=csv,noheader,nounits", "-lms", "200"],
                                         stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.t = threading.Thread(target=self._read, daemon=True)
            self.t.start()
        except Exception:
            self.proc = None
        return self

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def __exit__(self, *a):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()

    def summary(self):
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            parts = [p.strip() for p in ln.split(",")]
            if len(parts) < 7:
                continue
            try:
                sm.append(float(parts[0]))
                mx.append(float(parts[1]))
            except ValueError:
                continue
            for n, v in zip(names, parts[3:7]):
                if v.lower() == "active":
                    reasons.add(n)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"], "samples": 0}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "reasons": sorted(reasons),
                "samples": len(sm)}


# ------------------------------------------------------------------------------------------ oracle arm

def oracle_sample(wl, sc, n_tiles: int, n_layers: int, budget: int, device):
    """Time the CPU oracle on a bounded sample of the workload: Eq. 1 scoring + selection of
    n_tiles tiles, and the prefill of one sequence with `budget` vision tokens through n_layers
    layers.  Returns (seconds per tile, seconds per prefill token per layer, cores, sample text)."""
    from oracle import rift_oracle as O
    torch.set_num_threads(len(os.sched_getaffinity(0)))
    cores = torch.get_num_threads()
    dec = wl.decoder
    # a sample never exceeds the workload: small scenes and decoders are taken whole
    n_tiles = max(1, min(n_tiles, wl.scene.N))
    n_layers = max(1, min(n_layers, dec.n_layers))
    budget = max(0, min(budget, wl.scene.n_v))
    Xs = sc.X[:n_tiles].cpu()
    embed = sc.embed.cpu()
    t0 = time.perf_counter()
    t = O.query_embedding(embed, [sc.query_ids])
    B = O.background_embeddings(embed, sc.bg_ids)
    r64, V, s64 = O.score_scene(Xs, t, B)
    r32 = O.to_f32(r64)
    for i in range(n_tiles):
        O.top_b(r32[i], budget)
    t_tile = (time.perf_counter() - t0) / n_tiles
    sel = O.top_b(r32[0], budget)
    H0, cu, _ = O.pack(Xs, embed, [0], [sel], sc.sys_ids, sc.query_ids)
    L = H0.shape[0]
    layers = [W.make_layer(dec, l, device) for l in range(n_layers)]
    gf = W.make_final_norm(dec, device).cpu()
    t0 = time.perf_counter()
    h = H0.to(torch.float64)
    pos = torch.arange(L)
    for l in range(n_layers):
        h = O.decoder_layer(h, {k: v.cpu() for k, v in layers[l].items()}, dec, pos)
    O.rmsnorm(h, gf, dec.eps)
    t_tok_layer = (time.perf_counter() - t0) / (L * n_layers)
    text = (f"oracle on {n_tiles} of {wl.scene.N} tiles (scoring + top-b) and one {L}-token sequence through "
            f"{n_layers} of {dec.n_layers} layers (fp64), extrapolated linearly to the full query")
    return t_tile, t_tok_layer, cores, text


def oracle_tokens_per_s(wl, T, t_tile, t_tok_layer):
    step_s = wl.scene.N * t_tile + T * t_tok_layer * wl.decoder.n_layers
    return T / step_s, step_s


def expected_T(wl, sc, device):
    """Retained tokens of the query (from the oracle's own selection on the full scene)."""
    from oracle import rift_oracle as O
    if wl.policy.tau == 0.0 and wl.policy.C == (wl.scene.n_v,):
        return wl.scene.N * (wl.scene.S + wl.scene.n_v + wl.scene.Q)
    sel = O.select(sc.X.cpu(), sc.embed.cpu(), sc.query_ids, sc.bg_ids, wl.knn_m, wl.policy)
    return sum(wl.scene.S + b + wl.scene.Q for b in sel.budgets)


def run_reference(args, wl, ws, rank):
    if rank != 0:
        return
    dev = torch.device("cuda", 0) if torch.cuda.is_available() else torch.device("cpu")
    sc = W.make_scene(wl.scene, wl.decoder.vocab, dev)
    T = expected_T(wl, sc, dev)
    budget = min(wl.policy.C)
    times, vals = [], []
    for k in range(args.warmup + args.steps):
        t0 = time.perf_counter()
        t_tile, t_tok, cores, text = oracle_sample(wl, sc, 2, 2, budget, dev)
        v, _ = oracle_tokens_per_s(wl, T, t_tile, t_tok)
        if k >= args.warmup:
            times.append(time.perf_counter() - t0)
            vals.append(v)
    value = statistics.median(vals)
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * statistics.median(times),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {"workload": wl.name, "tiles": wl.scene.N, "retained_tokens_T": T},
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle",
                             "sample": "per step: " + text},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


# ------------------------------------------------------------------------------------------ main arm

L2_BYTES = 129 * 2 ** 20  # GB300 L2


def l2_note(x_bytes: int, w_bytes: int, flushed: bool) -> str:
    """How the timed steps keep L2 from carrying inputs over (the config's "l2" entry)."""
    sizes = "X %.2f GB, weights %.2f GB" % (x_bytes / 1e9, w_bytes / 1e9)
    if flushed:
        return "inputs fit in L2 (%s): L2 flushed between timed steps (a buffer of twice its size written outside the events)" % sizes
    return "inputs larger than L2 (%s)" % sizes

PROFILED_WORKLOAD = "rift400_7b"  # the workload of profiles/gemm_tc_traffic_rift400_7b.md


def gemm_traffic(workload: str):
    """DRAM bytes per GEMM launch from the committed ncu summary (one 7B layer at the 400-tile
    query's 23,819 retained rows: every GEMM shape of the query at its full size), if it was taken
    for this workload and on the current gemm_tc.cu (source hash match); otherwise None."""
    import hashlib
    import re
    if workload != PROFILED_WORKLOAD:
        return None
    prof = ROOT / "profiles" / "gemm_tc_traffic_rift400_7b.md"
    src = ROOT / "paper_2609_29029_gb300" / "csrc" / "gemm_tc.cu"
    if not prof.exists() or not src.exists():
        return None
    text = prof.read_text()
    h = re.search(r"source_sha256_16: ([0-9a-f]{16})", text)
    b = re.search(r"dram_bytes_per_launch: (\d+)", text)
    if not h or not b or hashlib.sha256(src.read_bytes()).hexdigest()[:16] != h.group(1):
        return None
    return int(b.group(1))


def select_latency(pipe, sc, q, bg, sy, steps: int, stream=None, batches: int = 5) -> float:
    """ms per query of scoring + selection + packing (the pre-prefill path): `batches` batches of
    `steps` queries enqueued back to back, each timed by events around it only, and the median
    batch reported (the first batch after a long power-capped prefill loop can run at a lower
    clock).  The stream is held by a short device-side sleep while the host enqueues a batch, so
    that the events time the device's work and not the host's launch rate (a query is ~15
    launches of well under a millisecond in all)."""
    st = stream if stream is not None else torch.cuda.current_stream()
    times = []
    for _ in range(batches):
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        if hasattr(torch.cuda, "_sleep"):
            with torch.cuda.stream(st):
                torch.cuda._sleep(int(2e6) * steps)  # ~1 ms of clock cycles per query at ~2 GHz
        e0.record(st)
        for _ in range(steps):
            pipe.run(sc.X, sc.embed, q, bg, sy, q, prefill=False, counts=False, stream=st)
        e1.record(st)
        torch.cuda.synchronize()
        times.append(e0.elapsed_time(e1) / steps)
    print("select latency per batch (ms/query): " + " ".join(f"{t:.4f}" for t in times), file=sys.stderr)
    return statistics.median(times)


def select_gather(n_kept: int, T: int, scene, x_elem: int, select_ms: float, pack_ms: float, hbm: float):
    """HBM roofline of selection + gather (prune/budgets, top-b, sequence offsets, packing) for one
    query: its algorithmic bytes -- the kept tiles' token scores r read, the selected token ids
    written and read back, the selected vision tokens and the prompt rows of the embedding table
    read, the packed rows written -- over the device time of the select and pack kernel classes."""
    if not (select_ms + pack_ms) > 0:
        return None
    sigma_b = T - n_kept * (scene.S + scene.Q)
    nbytes = (n_kept * scene.n_v * 4 + 2 * sigma_b * 4 + sigma_b * scene.d * x_elem
              + n_kept * (scene.S + scene.Q) * scene.d * 2 + T * scene.d * 2)
    ms = select_ms + pack_ms
    gbs = nbytes / (ms / 1e3) / 1e9
    return {"bytes_per_query": nbytes, "ms_per_query": ms, "achieved_gbs": gbs, "peak_gbs": hbm, "frac": gbs / hbm,
            "kernels": "select and pack classes: prune/budgets, top-b, sequence offsets, packing"}


def sweep(steps: int, warmup: int):
    """Scoring + selection + packing (no prefill) of the Rift policy over N tiles: per-step device
    time, per-kernel-class time, and the HBM rate of the token pass (N n_v d 2 bytes read)."""
    import __graft_entry__
    __graft_entry__.build()
    from paper_2609_29029_gb300 import ScenePipeline, abi
    dev = torch.device("cuda", 0)
    peaks = json.loads((ROOT / "MEASURED_PEAKS.json").read_text()) if (ROOT / "MEASURED_PEAKS.json").exists() else {}
    hbm = peaks.get("hbm_gbs", 6796.5)
    for N in W.SWEEP_N:
        wl = W.sweep_workload(N)
        s = wl.scene
        sc = W.make_scene(s, wl.decoder.vocab, dev)
        pipe = ScenePipeline(s.N, s.n_v, s.d, s.x_dtype, s.M, s.S, s.Q, wl.knn_m, wl.policy, device=dev)
        i32 = dict(dtype=torch.int32, device=dev)
        q, bg, sy = (torch.tensor(v, **i32) for v in (sc.query_ids, sc.bg_ids, sc.sys_ids))
        for _ in range(warmup):
            pipe.run(sc.X, sc.embed, q, bg, sy, q, prefill=False)
        torch.cuda.synchronize()
        ms = select_latency(pipe, sc, q, bg, sy, steps)
        n_kept, T = pipe.read_counts()
        # per-class breakdown in a separate pass (its events sit between the classes' launches)
        abi.profile_enable(True)
        for _ in range(steps):
            pipe.run(sc.X, sc.embed, q, bg, sy, q, prefill=False, counts=False)
        torch.cuda.synchronize()
        abi.profile_enable(False)
        prof = abi.profile_read()
        x_bytes = sc.X.numel() * sc.X.element_size()
        line = {"sweep": f"select+gather N={N}", "ms_per_query": ms,
                "kernels_ms": {k: round(v[0] / steps, 4) for k, v in prof.items() if v[1]},
                "kept_tiles": n_kept, "packed_rows": T, "x_bytes": x_bytes,
                "token_pass_lower_bound_ms": x_bytes / (hbm * 1e6),
                "select_gather": select_gather(n_kept, T, s, sc.X.element_size(), prof["select"][0] / steps,
                                               prof["pack"][0] / steps, hbm)}
        print(json.dumps(line), flush=True)
        del sc, pipe
        torch.cuda.empty_cache()


def shared_prefix_measure(pipe, sc, q, bg, sy, T, stream, steps):
    """The same scene query with the system prompt prefilled once and every sequence's suffix over
    its cache (rift_prefill_shared_prefix): same final hidden states, fewer rows prefilled.  Kept
    apart from the metric, whose token count it changes."""
    def one():
        return pipe.run_shared_prefix(sc.X, sc.embed, q, bg, sy, q, stream=stream)
    for _ in range(2):
        n_kept, T2 = one()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(steps):
        n_kept, T2 = one()
    e1.record(stream)
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1) / steps
    return {"ms_per_query": ms, "rows_prefilled": T2 + pipe.S, "rows_of_the_sequences": T,
            "retained_tokens_per_s_equivalent": T / (ms / 1e3), "note": "system prompt prefilled once; "
            "the suffixes attend to its cache"}


def decode_measure(pipe, dm, sc, dec, n_kept, T, stream, steps):
    """The first decode step after the prefill (Section 2.1), timed on its own: the prefill runs
    once more writing its KV cache, then `steps` decode steps of one seeded token per retained
    tile.  Reported beside the prefill metric (not part of it), with its HBM roofline: every
    weight, the output matrix and the whole KV cache are read once per step."""
    from paper_2609_29029_gb300 import abi
    dev = sc.X.device
    d = dec.d
    pipe.run(sc.X, sc.embed, *(torch.tensor(v, dtype=torch.int32, device=dev)
                               for v in (sc.query_ids, sc.bg_ids, sc.sys_ids, sc.query_ids)),
             prefill=False, stream=stream)
    kv = torch.empty(dec.n_layers, 2, T, d, dtype=torch.float16, device=dev)
    last = torch.empty(n_kept, dec.vocab, dtype=torch.float32, device=dev)
    pipe.prefill(stream, kv_out=kv, last_logits=last, counts=(n_kept, T))
    key = rng.stream_key(0, rng.stream_id("bench-decode"))
    ids = torch.tensor([rng.hash_u32_int(key, i) % dec.vocab for i in range(n_kept)], dtype=torch.int32, device=dev)
    hid = torch.empty(n_kept, d, dtype=torch.bfloat16, device=dev)
    lg = torch.empty(n_kept, dec.vocab, dtype=torch.float32, device=dev)
    max_len = pipe.max_len + 1
    need = abi.decode_workspace_bytes(dm.struct, n_kept, max_len)
    ws = torch.empty(need, dtype=torch.uint8, device=dev)

    def one():
        abi.decode_step(dm.struct, kv, T, pipe.cu, n_kept, max_len, ids, sc.embed, sc.embed.shape[0], hid, None, lg,
                        ws, need, stream)

    for _ in range(3):
        one()
    abi.sync_status(stream)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    if hasattr(torch.cuda, "_sleep"):  # hold the stream while the host enqueues (see select_latency)
        with torch.cuda.stream(stream):
            torch.cuda._sleep(int(4e6) * steps)
    e0.record(stream)
    for _ in range(steps):
        one()
    e1.record(stream)
    torch.cuda.synchronize()
    abi.sync_status(stream)
    ms = e0.elapsed_time(e1) / steps
    abi.profile_enable(True)  # per-class breakdown, in a separate untimed pass
    for _ in range(steps):
        one()
    torch.cuda.synchronize()
    abi.profile_enable(False)
    breakdown = {k: round(v[0] / steps, 3) for k, v in abi.profile_read().items() if v[1]}
    weights = dec.n_layers * dec.params_per_layer * 2 + dec.vocab * d * 2
    kv_bytes = dec.n_layers * 2 * T * d * 2
    peaks = json.loads((ROOT / "MEASURED_PEAKS.json").read_text()) if (ROOT / "MEASURED_PEAKS.json").exists() else {}
    hbm = peaks.get("hbm_gbs", 6800.0)
    gbs = (weights + kv_bytes) / (ms / 1e3) / 1e9
    del kv
    torch.cuda.empty_cache()
    return {"ms": ms, "tokens_per_s": n_kept / (ms / 1e3), "sequences": n_kept, "cached_rows": T,
            "kernels_ms": breakdown, "algorithmic_bytes": weights + kv_bytes, "achieved_gbs": gbs, "peak_gbs": hbm, "frac_hbm": gbs / hbm,
            "bound": "hbm", "inputs": "seeded token ids; KV cache from the prefill of the same query"}


def batch_measure(dm, dec, base, stream, steps, B=8, N=64):
    """Several scene queries per prefill (rift_pack_ragged_at): B queries over B different
    N-tile scenes (the small end of the paper's 64..400-tile scenes), timed batched against one
    query at a time.  Reported beside the metric."""
    from dataclasses import replace
    from paper_2609_29029_gb300 import ScenePipeline
    dev = torch.device("cuda", torch.cuda.current_device())
    i32 = dict(dtype=torch.int32, device=dev)
    spec = replace(base.scene, N=N)
    queries = []
    for b in range(B):
        sc = W.make_scene(replace(spec, seed=100 + b), dec.vocab, dev)
        q = torch.tensor(sc.query_ids, **i32)
        queries.append((sc.X, sc.embed, q, torch.tensor(sc.bg_ids, **i32), torch.tensor(sc.sys_ids, **i32), q))
    pipe = ScenePipeline(N, spec.n_v, spec.d, spec.x_dtype, spec.M, spec.S, spec.Q, base.knn_m, base.policy,
                         model=dm, device=dev)
    res = pipe.run_batch(queries, stream=stream)
    for qq in queries:
        pipe.run(*qq, stream=stream)
    torch.cuda.synchronize()
    rows = sum(r[1] for r in res)

    def timed(fn):
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(steps):
            fn()
        e1.record(stream)
        torch.cuda.synchronize()
        return e0.elapsed_time(e1) / steps

    ms_b = timed(lambda: pipe.run_batch(queries, stream=stream))
    ms_1 = timed(lambda: [pipe.run(*qq, stream=stream, counts=False) for qq in queries])
    del queries, pipe
    torch.cuda.empty_cache()
    return {"queries": B, "tiles_per_scene": N, "retained_rows": rows,
            "batched_ms": ms_b, "one_at_a_time_ms": ms_1,
            "batched_scene_queries_per_s": B / (ms_b / 1e3), "one_at_a_time_scene_queries_per_s": B / (ms_1 / 1e3),
            "batched_tokens_per_s": rows / (ms_b / 1e3)}


def kernel_case(name: str):
    """Small cases for ncu captures: inputs larger than L2, about 1 GB on the device."""
    import __graft_entry__
    __graft_entry__.build()
    from paper_2609_29029_gb300 import DeviceModel, ScenePipeline, abi
    dev = torch.device("cuda", 0)
    if name in ("prefill", "prefill_full"):
        dec = W.DecoderShape(n_layers=1, d=4096, n_heads=32, head_dim=128, ffn=11008, vocab=32000)
        dm = DeviceModel(dec, [W.make_layer(dec, 0, dev)], W.make_final_norm(dec, dev), dev)
        # prefill_full: the retained length mix of the 400-tile query (63 tiles at b = 288, 9 at
        # 144, 1 at 72, each with the 35 system and 24 query rows): every GEMM at its full M
        lens = [341] * 12 if name == "prefill" else [347] * 63 + [203] * 9 + [131]
        T = sum(lens)
        from synth import rng
        H0 = rng.normal_f32(0, rng.stream_id("case"), T * dec.d, dev).view(T, dec.d).to(torch.bfloat16)
        cu = torch.tensor([0] + [sum(lens[:i + 1]) for i in range(len(lens))], dtype=torch.int32, device=dev)
        pos = torch.cat([torch.arange(L, dtype=torch.int32, device=dev) for L in lens])
        need = abi.prefill_workspace_bytes(dm.struct, T, len(lens), 635)
        ws = torch.empty(need, dtype=torch.uint8, device=dev)
        for _ in range(3):
            hid = H0.clone()
            abi.prefill_layers(dm.struct, hid, T, cu, len(lens), 635, pos, ws, need)
        abi.sync_status()
    elif name == "attention":
        # the attention of one 7B-shaped layer over equal-length sequences: time per length
        H, HD = 32, 128
        d = H * HD
        peaks = json.loads((ROOT / "MEASURED_PEAKS.json").read_text()) if (ROOT / "MEASURED_PEAKS.json").exists() else {}
        hbm = peaks.get("hbm_gbs", 6796.5)
        flush = torch.empty(2 * L2_BYTES, dtype=torch.uint8, device=dev)
        from synth import rng
        for L in (131, 203, 256, 347, 512, 1024, 2048, 4096):
            n = max(1, 23819 // L)
            T = n * L
            qkv = rng.normal_f32(0, rng.stream_id("case-attn", L), T * 3 * d, dev).view(T, 3 * d).to(torch.float16)
            out = torch.empty(T, d, dtype=torch.float16, device=dev)
            cu = torch.tensor([i * L for i in range(n + 1)], dtype=torch.int32, device=dev)
            need = abi.attention_workspace_bytes(T, n)
            ws = torch.empty(need, dtype=torch.uint8, device=dev)
            for _ in range(3):
                abi.attention_varlen(qkv, T, cu, n, H, HD, out, ws, need)
            times = []
            for _ in range(10):
                flush.fill_(1)
                e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                e0.record()
                abi.attention_varlen(qkv, T, cu, n, H, HD, out, ws, need)
                e1.record()
                torch.cuda.synchronize()
                times.append(e0.elapsed_time(e1))
            ms = statistics.median(times)
            blocks = n * H * sum(-(-min(L, 128 * b + 128) // 64) for b in range(-(-L // 128)))
            print(json.dumps({"L": L, "sequences": n, "T": T, "us": round(1e3 * ms, 1), "kv_blocks": blocks,
                              "us_per_block_per_cta_slot": round(1e3 * ms * 2 * 152 / blocks, 3),
                              "of_hbm_floor": round(8 * d * T / (ms / 1e3) / (hbm * 1e9), 3)}), flush=True)
            del qkv, out, ws
        abi.sync_status()
    elif name == "merge":
        # the 400-tile scene's selection with Stage 2's merge, three times
        wl = W.RIFT400_MERGE
        s = wl.scene
        sc = W.make_scene(s, wl.decoder.vocab, dev)
        pipe = ScenePipeline(s.N, s.n_v, s.d, s.x_dtype, s.M, s.S, s.Q, wl.knn_m, wl.policy, device=dev)
        i32 = dict(dtype=torch.int32, device=dev)
        for _ in range(3):
            pipe.select(sc.X, sc.embed, torch.tensor(sc.query_ids, **i32), torch.tensor(sc.bg_ids, **i32))
            pipe.merge(sc.X)
        abi.sync_status()
    elif name == "decode":
        # 4 layers of the 7B shape, 73 sequences of 130..635 cached rows (about the retained set
        # of the 400-tile query), a random fp16 KV cache: three decode steps
        dec = W.DecoderShape(n_layers=4, d=4096, n_heads=32, head_dim=128, ffn=11008, vocab=32000)
        dm = DeviceModel(dec, [W.make_layer(dec, l, dev) for l in range(dec.n_layers)], W.make_final_norm(dec, dev),
                         dev, lm_head=W.make_lm_head(dec, dev))
        lens = [35 + 24 + (72, 144, 288, 432, 576)[i % 5] for i in range(73)]
        T, n = sum(lens), len(lens)
        cu = torch.tensor([0] + [sum(lens[:i + 1]) for i in range(n)], dtype=torch.int32, device=dev)
        from synth import rng
        kv = rng.normal_f32(0, rng.stream_id("case-kv"), dec.n_layers * 2 * T * dec.d, dev).to(torch.float16)
        embed = rng.normal_f32(0, rng.stream_id("case-embed"), 1024 * dec.d, dev).view(1024, dec.d).to(torch.bfloat16)
        ids = torch.arange(n, dtype=torch.int32, device=dev)
        hid = torch.empty(n, dec.d, dtype=torch.bfloat16, device=dev)
        lg = torch.empty(n, dec.vocab, dtype=torch.float32, device=dev)
        need = abi.decode_workspace_bytes(dm.struct, n, 636)
        ws = torch.empty(need, dtype=torch.uint8, device=dev)
        for _ in range(3):
            abi.decode_step(dm.struct, kv, T, cu, n, 636, ids, embed, 1024, hid, None, lg, ws, need)
        abi.sync_status()
    else:
        wl = W.sweep_workload(64)
        s = wl.scene
        sc = W.make_scene(s, wl.decoder.vocab, dev)
        pipe = ScenePipeline(s.N, s.n_v, s.d, s.x_dtype, s.M, s.S, s.Q, wl.knn_m, wl.policy, device=dev)
        i32 = dict(dtype=torch.int32, device=dev)
        for _ in range(3):
            pipe.select(sc.X, sc.embed, torch.tensor(sc.query_ids, **i32), torch.tensor(sc.bg_ids, **i32))
        abi.sync_status()
    print(f"kernel case {name}: ok")


def main():
    args = parse()
    if args.ncu_summary:
        print(ncu_summary(args.ncu_summary))
        return
    if args.kernel_case:
        kernel_case(args.kernel_case)
        return
    if args.sweep:
        sweep(args.steps, max(args.warmup, 1))
        return
    ws, rank, local = dist_setup()
    wl = W.WORKLOADS[args.workload]
    if args.impl == "reference":
        run_reference(args, wl, ws, rank)
        return
    import __graft_entry__
    __graft_entry__.build()
    from paper_2609_29029_gb300 import DeviceModel, ScenePipeline, abi

    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    s, dec = wl.scene, wl.decoder
    sc = W.make_scene(s, dec.vocab, dev)
    layers = [W.make_layer(dec, l, dev) for l in range(dec.n_layers)]
    dm = DeviceModel(dec, layers, W.make_final_norm(dec, dev), dev, lm_head=W.make_lm_head(dec, dev))
    del layers
    pipe = ScenePipeline(s.N, s.n_v, s.d, s.x_dtype, s.M, s.S, s.Q, wl.knn_m, wl.policy, model=dm, device=dev)
    i32 = dict(dtype=torch.int32, device=dev)
    q = torch.tensor(sc.query_ids, **i32)
    bg = torch.tensor(sc.bg_ids, **i32)
    sy = torch.tensor(sc.sys_ids, **i32)
    stream = torch.cuda.current_stream()

    def step(X, counts=True):
        return pipe.run(X, sc.embed, q, bg, sy, q, stream=stream, counts=counts)

    for _ in range(max(args.warmup, 1)):
        n_kept, T = step(sc.X)
    torch.cuda.synchronize()

    # ---- timed region: inputs resident in HBM.  When the query's inputs (tokens and weights)
    # could stay in L2 between steps, each step is timed by its own events and L2 is flushed
    # between steps (outside the events) by writing a buffer twice its size.
    in_bytes = sc.X.numel() * sc.X.element_size() + dec.n_layers * dec.params_per_layer * 2
    flush = None
    if in_bytes < 2 * L2_BYTES:
        flush = torch.empty(2 * L2_BYTES // 4, dtype=torch.float32, device=dev)
    barrier(ws)
    torch.cuda.synchronize()
    abi.profile_enable(True)
    l0 = abi.launch_count()
    with ClockSampler(local) as clk:
        if flush is None:
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            for _ in range(args.steps):  # whole queries enqueued back to back: no host read-back
                step(sc.X, counts=False)
            e1.record(stream)
            torch.cuda.synchronize()
            ms = e0.elapsed_time(e1)
            n_kept, T = pipe.read_counts(stream)
        else:
            evs = []
            for _ in range(args.steps):
                flush.fill_(1.0)
                e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                e0.record(stream)
                step(sc.X, counts=False)
                e1.record(stream)
                evs.append((e0, e1))
            torch.cuda.synchronize()
            ms = sum(a.elapsed_time(b) for a, b in evs)
            n_kept, T = pipe.read_counts(stream)
    launches = abi.launch_count() - l0
    abi.profile_enable(False)
    prof = abi.profile_read()
    barrier(ws)
    value, ms_max = job_throughput(float(T * args.steps), ms, ws)
    # the pre-prefill path alone (scoring, selection, packing), without the profiler's events
    # between its classes
    sel_ms = select_latency(pipe, sc, q, bg, sy, args.steps, stream)

    # ---- end to end: host buffers.  Every step copies its inputs (the scene's vision tokens and
    # the query's id lists) from pinned host memory and reads its result (the final hidden states)
    # back; the decoder's weights and embedding table are model state, resident like the other
    # weights.  As a stream of scene queries would be served, the next step's inputs are copied on
    # one stream into the other of two input buffers, and each result is copied out on another
    # stream while the next query computes (two pipelines, so a result is never overwritten
    # before it has been read out).  The timed region ends when the last result is on the host.
    X_host = sc.X.cpu().pin_memory()
    ids_host = [torch.tensor(v, dtype=torch.int32).pin_memory() for v in (sc.query_ids, sc.bg_ids, sc.sys_ids)]
    bufs = [dict(X=torch.empty_like(sc.X), ids=[torch.empty_like(h, device=dev) for h in ids_host]) for _ in range(2)]
    pipes = [pipe, ScenePipeline(s.N, s.n_v, s.d, s.x_dtype, s.M, s.S, s.Q, wl.knn_m, wl.policy, model=dm,
                                 device=dev)]
    out_host = [torch.empty(T, s.d, dtype=torch.bfloat16).pin_memory() for _ in range(2)]
    copy_stream = torch.cuda.Stream(device=dev)
    d2h_stream = torch.cuda.Stream(device=dev)

    def h2d(buf):
        with torch.cuda.stream(copy_stream):
            buf["X"].copy_(X_host, non_blocking=True)
            for hdst, hsrc in zip(buf["ids"], ids_host):
                hdst.copy_(hsrc, non_blocking=True)
            ev = torch.cuda.Event()
            ev.record(copy_stream)
        return ev

    def e2e_steps(n):
        Te = 0
        ready = h2d(bufs[0])
        read_out = [None, None]  # per pipeline: its last result copy
        for k in range(n):
            buf, p = bufs[k % 2], pipes[k % 2]
            stream.wait_event(ready)
            if read_out[k % 2] is not None:  # this pipeline's previous result is on the host
                stream.wait_event(read_out[k % 2])
            if k + 1 < n:  # the other input buffer is free: its last reader (step k - 1) has finished
                nxt = torch.cuda.Event()
                nxt.record(stream)
                copy_stream.wait_event(nxt)
                ready = h2d(bufs[(k + 1) % 2])
            p.run(buf["X"], sc.embed, buf["ids"][0], buf["ids"][1], buf["ids"][2], buf["ids"][0], stream=stream,
                  counts=False)
            # the result's size: wait for this query's packing only (its prefill stays queued)
            nk, Te = p.counts()
            done = torch.cuda.Event()
            done.record(stream)
            d2h_stream.wait_event(done)
            with torch.cuda.stream(d2h_stream):
                out_host[k % 2][:Te].copy_(p.packed[:Te], non_blocking=True)
                ev = torch.cuda.Event()
                ev.record(d2h_stream)
            read_out[k % 2] = ev
        for ev in read_out:
            if ev is not None:
                stream.wait_event(ev)
        return Te

    e2e_steps(2)  # warm-up: first touch of the buffers and of the second pipeline's workspace
    torch.cuda.synchronize()
    barrier(ws)
    torch.cuda.synchronize()
    f0, f1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with ClockSampler(local) as clk_e2e:
        f0.record(stream)
        Te = e2e_steps(args.e2e_steps)
        f1.record(stream)
        torch.cuda.synchronize()
    e2e_val, _ = job_throughput(float(Te * args.e2e_steps), f0.elapsed_time(f1), ws)
    h2d_bytes = X_host.numel() * X_host.element_size() + sum(h.numel() * 4 for h in ids_host)
    del pipes, bufs, out_host, X_host
    torch.cuda.empty_cache()
    d2h = Te * s.d * 2 + 8
    decode = None if args.no_decode else decode_measure(pipe, dm, sc, dec, n_kept, T, stream, args.steps)
    shared = None if args.no_shared_prefix else shared_prefix_measure(pipe, sc, q, bg, sy, T, stream, args.steps)
    batch = None if args.no_batch else batch_measure(dm, dec, wl, stream, max(2, args.steps // 2))

    if rank != 0:
        return
    # ---- roofline of the dominant kernel (the prefill GEMM) from the live event timing
    peaks = json.loads((ROOT / "MEASURED_PEAKS.json").read_text()) if (ROOT / "MEASURED_PEAKS.json").exists() else {}
    peak = peaks.get("bf16_tflops_sustained", 1700.0)
    gemm_ms, gemm_n = prof["gemm"]
    gemm_flops = args.steps * T * dec.linear_flops_per_token
    achieved = gemm_flops / (gemm_ms / 1e3) / 1e12 if gemm_ms > 0 else None
    traffic = gemm_traffic(wl.name)
    peak_burst = peaks.get("bf16_tflops", 1887.6)
    per_step = {k: round(v[0] / args.steps, 3) for k, v in prof.items()}
    x_bytes = sc.X.numel() * sc.X.element_size()
    hbm = peaks.get("hbm_gbs", 6796.5)
    sigma_b = T - n_kept * (s.S + s.Q)
    sel_gather = select_gather(n_kept, T, s, sc.X.element_size(), prof["select"][0] / args.steps,
                               prof["pack"][0] / args.steps, hbm)

    cpu = None
    if not args.no_cpu_baseline and ws == 1:
        t_tile, t_tok, cores, text = oracle_sample(wl, sc, 8, 4, int(round((T / max(n_kept, 1)) - s.S - s.Q)), dev)
        v, step_s = oracle_tokens_per_s(wl, T, t_tile, t_tok)
        cpu = {"value": v, "unit": UNIT, "cores": cores, "kind": "oracle", "sample": text,
               "extrapolated_step_s": step_s}

    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": ws, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": ms_max / args.steps, "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "f16", "data": "synthetic",
        "config": {"workload": wl.name, "tiles": s.N, "tokens_per_tile": s.n_v, "d": s.d,
                   "decoder": f"{dec.n_layers}x{dec.d} LLaMA/Vicuna-7B shape, random init",
                   "kept_tiles": n_kept, "retained_tokens_T": T,
                   "mean_budget_frac": round((T / max(n_kept, 1) - s.S - s.Q) / s.n_v, 4),
                   "parallelism": f"replicas x{ws}" if ws > 1 else "single GPU",
                   "l2": l2_note(sc.X.numel() * sc.X.element_size(), dec.n_layers * dec.params_per_layer * 2,
                                 flush is not None)},
        "scene_queries_per_s": 1e3 * args.steps / ms_max,
        "vision_tokens_per_s": value * sigma_b / max(T, 1),
        "select_latency_ms": sel_ms,
        "select_latency_floor_ms": x_bytes / (hbm * 1e6),
        "select_gather": sel_gather,
        "kernels_ms_per_step": per_step,
        "roofline": {"bound": "tensor", "kernel": "prefill GEMM", "achieved": achieved, "peak": peak,
                     "unit": "TFLOP/s", "frac": (achieved / peak) if achieved else None, "traffic": traffic,
                     "peak_source": "MEASURED_PEAKS.json bf16_tflops_sustained (of measured)",
                     "peak_burst": peak_burst, "frac_burst": (achieved / peak_burst) if achieved else None,
                     "launches": gemm_n},
        "cpu_baseline": cpu,
        "e2e": {"value": e2e_val, "unit": UNIT, "h2d_bytes_per_step": h2d_bytes, "d2h_bytes_per_step": d2h,
                "steps": args.e2e_steps, "clocks": clk_e2e.summary(),
                "copies": "in: vision tokens and id lists (pinned host); out: final hidden states and the two "
                          "counts; embedding table and weights resident"},
        "decode_step": decode,
        "shared_prefix": shared,
        "batch": batch,
        "gpu_launches": launches,
        "clocks": clk.summary(),
    }
    print(json.dumps(line), flush=True)


if __name__ == "__main__":
    main()
