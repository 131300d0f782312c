"""One scene query sharded over gloo ranks on the CPU (no GPU).

Each rank holds a contiguous shard of the tiles and runs the sharding protocol of
paper_2609_29029_gb300.shard with the oracle as its per-rank engine: its own scores, an all-gather
of the tile embeddings and raw scores for the kNN smoothing (Appendix B Step 2), an all-reduce of
the smoothed scores' (min, max) for the per-scene min-max (Section 2.3 Stage 1), its own
selection, then a cost-balanced all-to-all of the packed sequences and the prefill of the
sequences it was given.  The union over the ranks must equal the oracle's single-rank query bit
for bit: neighbour sets, smoothed scores, u, kept tiles, budgets, selected tokens, packed rows and
final hidden states.  One test has a rank leave between two queries: the others see it through
the store, form a group of the survivors and re-shard.
"""
import os
import sys
from pathlib import Path

import numpy as np
import pytest
import torch
import torch.multiprocessing as mp

ROOT = Path(__file__).resolve().parent.parent
TESTS = Path(__file__).resolve().parent


def _scene(name):
    import parity as P
    from synth import workloads as W
    wl = {P.SMALL24.name: P.SMALL24, P.RAGGED.name: P.RAGGED}[name]
    sc = W.make_scene(wl.scene, wl.decoder.vocab)
    layers = [W.make_layer(wl.decoder, l) for l in range(wl.decoder.n_layers)]
    return wl, sc, layers, W.make_final_norm(wl.decoder)


def _engine(wl, sc, layers, gf, lo, hi):
    from shard_oracle import OracleShardEngine
    return OracleShardEngine(sc.X[lo:hi], sc.embed, sc.query_ids, sc.bg_ids, sc.sys_ids, wl.knn_m, wl.policy,
                             get_layer=lambda l: layers[l], g_final=gf, dec=wl.decoder)


def _pack_result(res):
    # plain numpy arrays: a queue hands torch tensors over through shared memory that dies with
    # the rank's process
    return dict(kept=res.kept, budgets=res.budgets, sel=res.sel, u=res.u.numpy().copy(),
                tile_s=res.tile_s.numpy().copy(), nbr=res.nbr.numpy().copy(), seq_tiles=res.seq_tiles,
                cu=res.cu, rows=res.rows.numpy().copy(), bounds=res.bounds)


def _rank(rank, ws, port, name, leave_after, out):
    code = 0
    try:
        _rank_body(rank, ws, port, name, leave_after, out)
    except BaseException:
        import traceback
        out.put((rank, -1, traceback.format_exc()))
        code = 1
    out.close()
    out.join_thread()  # the queue's feeder thread has written everything
    os._exit(code)  # the process group of a departed rank is not torn down collectively


def _rank_body(rank, ws, port, name, leave_after, out):
    sys.path[:0] = [str(ROOT), str(TESTS)]
    import torch.distributed as dist
    from paper_2609_29029_gb300 import shard
    store = dist.TCPStore("127.0.0.1", port, ws, rank == 0, wait_for_workers=True)
    dist.init_process_group("gloo", store=store, rank=rank, world_size=ws)
    wl, sc, layers, gf = _scene(name)
    mem = shard.Membership(store, rank, ws, timeout=60.0)
    steps = 1 if leave_after is None else 2
    for step in range(steps):
        if leave_after is not None and step > 0 and rank == leave_after:
            mem.leave()  # between queries: nothing of this rank is in flight
            out.put((rank, step, None))
            break
        group, r, R = mem.group(step)
        b = shard.shard_bounds(wl.scene.N, R)
        eng = _engine(wl, sc, layers, gf, b[r], b[r + 1])
        res = shard.run_group(shard.sharded_query(eng, r, R, wl.scene.N, dec=wl.decoder), group)
        out.put((rank, step, _pack_result(res)))
    # rank 0 hosts the store: it stays until every rank has finished with it
    store.add("rift_done", 1)
    if rank == 0:
        import time
        t0 = time.monotonic()
        while store.add("rift_done", 0) < ws and time.monotonic() - t0 < 60:
            time.sleep(0.01)


def _run(name, ws, port, leave_after=None):
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    procs = [ctx.Process(target=_rank, args=(r, ws, port, name, leave_after, q)) for r in range(ws)]
    for p in procs:
        p.start()
    # one result per rank and query, and the leaving rank's notice
    n_msgs = ws if leave_after is None else ws + (ws - 1) + 1
    msgs = []
    try:
        while len(msgs) < n_msgs:
            m = q.get(timeout=300)
            assert m[1] != -1, f"rank {m[0]} failed:\n{m[2]}"
            msgs.append(m)
        for p in procs:
            p.join(timeout=120)
            assert p.exitcode == 0
    finally:
        for p in procs:  # a failed rank leaves the others waiting in a collective
            if p.is_alive():
                p.kill()
    return msgs


def _check_union(name, results):
    """The ranks' results of one query against the oracle's whole-scene query."""
    from oracle import rift_oracle as O
    wl, sc, layers, gf = _scene(name)
    sel = O.select(sc.X, sc.embed, sc.query_ids, sc.bg_ids, wl.knn_m, wl.policy)
    R = len(results)  # in rank order within the query's group: shard r is bounds[r] .. bounds[r + 1]
    bounds = results[0]["bounds"]
    assert len(bounds) == R + 1 and all(res["bounds"] == bounds for res in results)
    kept, budgets, toks, u, st, nbr = [], [], [], [], [], []
    for r in range(R):
        res = results[r]
        kept += res["kept"]
        budgets += res["budgets"]
        toks += res["sel"]
        u.append(res["u"])
        st.append(res["tile_s"])
        nbr.append(res["nbr"])
    assert kept == sel.kept
    assert budgets == sel.budgets
    assert toks == sel.sel
    assert np.concatenate(u).view(np.uint32).tolist() == sel.u.view(np.uint32).tolist()
    assert np.concatenate(st).view(np.uint32).tolist() == sel.s_tilde.view(np.uint32).tolist()
    assert np.array_equal(np.concatenate(nbr), sel.nbr)
    # every kept tile's sequence was prefilled by exactly one rank, with the oracle's packed rows
    # and final hidden states
    H0, cu, _ = O.pack(sc.X, sc.embed, sel.kept, sel.sel, sc.sys_ids, sc.query_ids)
    seen = []
    for res in results:
        for j, t in enumerate(res["seq_tiles"]):
            k = sel.kept.index(t)
            rows = torch.from_numpy(res["rows"][res["cu"][j]:res["cu"][j + 1]])
            ref = O.prefill_sequence(H0[cu[k]:cu[k + 1]], lambda l: layers[l], gf, wl.decoder)
            assert torch.equal(rows, ref)
            seen.append(t)
    assert sorted(seen) == sel.kept
    # the prefill work is balanced: no rank has more than the largest sequence above the mean
    costs = [sum(cu[sel.kept.index(t) + 1] - cu[sel.kept.index(t)] for t in res["seq_tiles"]) for res in results]
    assert max(costs) - min(costs) <= max(cu[k + 1] - cu[k] for k in range(len(sel.kept)))


@pytest.mark.parametrize("name,ws,port", [("small24_f32", 2, 29621), ("ragged40_bf16", 3, 29622)])
def test_sharded_query_equals_single_rank_oracle(name, ws, port):
    # ragged40 over 3 ranks: shards of 13, 13 and 14 tiles
    msgs = _run(name, ws, port)
    results = [m[2] for m in sorted(msgs, key=lambda m: m[0])]
    _check_union(name, results)


def test_rank_leaving_between_queries_reshards(tmp_path):
    # three ranks answer one query; rank 2 then leaves; ranks 0 and 1 re-shard the scene over
    # themselves (12 + 12 tiles instead of 8 + 8 + 8) and answer the next query
    msgs = _run("small24_f32", 3, 29623, leave_after=2)
    first = [m[2] for m in sorted(msgs, key=lambda m: m[0]) if m[1] == 0]
    second = [m[2] for m in sorted(msgs, key=lambda m: m[0]) if m[1] == 1 and m[2] is not None]
    left = [m for m in msgs if m[1] == 1 and m[2] is None]
    assert len(first) == 3 and len(second) == 2 and [m[0] for m in left] == [2]
    assert first[0]["bounds"] == [0, 8, 16, 24] and second[0]["bounds"] == [0, 12, 24]
    _check_union("small24_f32", first)
    _check_union("small24_f32", second)


def test_rebalance_is_deterministic_and_balanced():
    from paper_2609_29029_gb300 import shard
    from synth import workloads as W
    dec = W.LLAVA7B
    seqs = [(t, L) for t, L in zip(range(0, 40, 3), [347, 131, 203, 347, 347, 635, 131, 203, 347, 490, 347, 203, 347, 635])]
    a = shard.rebalance(seqs, 3, dec)
    assert a == shard.rebalance(list(reversed(seqs)), 3, dec)  # order of the gathered list does not matter
    assert sorted(t for part in a for t in part) == [t for t, _ in seqs]
    cost = [sum(shard.sequence_cost(dict(seqs)[t], dec) for t in part) for part in a]
    assert max(cost) - min(cost) <= shard.sequence_cost(635, dec)
    assert shard.shard_bounds(40, 3) == [0, 13, 26, 40]
    with pytest.raises(ValueError):
        shard.shard_bounds(2, 3)
