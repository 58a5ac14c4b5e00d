"""The N > 1 path on CPU (gloo, world size 2, 127.0.0.1).

Data parallelism shards the batch by sequence; masks are keyed by the global
sequence index, so each shard draws exactly its slice of the full batch's
masks, computes its sequences independently, and the only exchange is the
all-reduce (sum) of the weight gradients.  Checked with the oracle: shard
outputs equal the full-batch slices, the all-reduced shard gradients equal
the full-batch gradients, for per-sequence masks and for per-token masks
(keyed by the global token index).  Also the benchmark's max-over-ranks step
time."""

import os
import socket

import numpy as np
import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

from paper_2609_05275_gb300 import synth


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    p = s.getsockname()[1]
    s.close()
    return p


def _worker(rank, world, port, q):
    import sys
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    sys.path.insert(0, root)
    sys.path.insert(0, os.path.join(root, "tests"))
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        from oracle import masks as OM, schedule as OS, stack as OK
        import bench

        cfg = dict(synth.CONFIGS["tiny"], B=4, L=2)
        B = cfg["B"]
        Bs = B // world
        sched = dict(dist="explicit", p_explicit=[0.3, 0.6], time="const")
        rates = OS.layer_rates(sched, cfg["L"], 0)
        thr = [OS.drop_threshold(p) for p in rates]
        scales = [OS.residual_scale(p) for p in rates]
        full_mask = OM.draw_masks(5, 3, thr, B)
        mask = OM.draw_masks(5, 3, thr, Bs, b_offset=rank * Bs)
        ok_mask = bool((mask == full_mask[:, rank * Bs:(rank + 1) * Bs]).all())
        # per-shard granularity: each rank draws for its whole shard, keyed by its first global sequence
        shard = OM.draw_masks(5, 3, thr, Bs, OM.PER_SHARD, b_offset=rank * Bs)
        ok_mask = ok_mask and bool((shard == full_mask[:, rank * Bs:rank * Bs + 1]).all())
        # per-token granularity: a shard's tokens are the global tokens of its sequences
        S = cfg["S"]
        full_tok = OM.draw_masks(5, 3, thr, B, OM.PER_TOKEN, S=S)
        tok = OM.draw_masks(5, 3, thr, Bs, OM.PER_TOKEN, b_offset=rank * Bs, S=S)
        ok_mask = ok_mask and bool((tok == full_tok[:, rank * Bs:(rank + 1) * Bs]).all())
        layers = [{n: v.double().numpy() for n, v in W.items()} for W in synth.stack_weights(cfg, seed=0)]
        x = synth.activations(cfg, seed=0, B=B).double().numpy()
        dy = synth.upstream_grad(cfg, B=B).double().numpy()
        sl = slice(rank * Bs, (rank + 1) * Bs)
        out, caches = OK.stack_forward(x[sl], layers, cfg, mask, scales)
        dX, grads = OK.stack_backward(dy[sl], layers, cfg, mask, scales, caches)
        summed = {}
        for l in range(cfg["L"]):
            for n, g in grads[l].items():
                t = torch.from_numpy(g.copy())
                dist.all_reduce(t, op=dist.ReduceOp.SUM)
                summed[(l, n)] = t.numpy()
        # the same with per-token masks
        tout, tc = OK.stack_forward(x[sl], layers, cfg, tok, scales, per_token=True)
        tdX, tgrads = OK.stack_backward(dy[sl], layers, cfg, tok, scales, tc, per_token=True)
        tsummed = {}
        for l in range(cfg["L"]):
            for n, g in tgrads[l].items():
                t = torch.from_numpy(g.copy())
                dist.all_reduce(t, op=dist.ReduceOp.SUM)
                tsummed[(l, n)] = t.numpy()
        ms = bench.max_over_ranks(10.0 + rank, world, device="cpu")
        res = dict(rank=rank, ok_mask=ok_mask, ms=ms)
        if rank == 0:
            fout, fc = OK.stack_forward(x, layers, cfg, full_mask, scales)
            fdX, fg = OK.stack_backward(dy, layers, cfg, full_mask, scales, fc)
            res["out_ok"] = bool(np.array_equal(out, fout[sl]) and np.array_equal(dX, fdX[sl]))
            res["grad_err"] = max(float(np.abs(summed[(l, n)] - fg[l][n]).max() / (np.abs(fg[l][n]).max() + 1e-30))
                                  for l in range(cfg["L"]) for n in fg[l])
            gout, gc = OK.stack_forward(x, layers, cfg, full_tok, scales, per_token=True)
            gdX, gg = OK.stack_backward(dy, layers, cfg, full_tok, scales, gc, per_token=True)
            res["tok_out_ok"] = bool(np.array_equal(tout, gout[sl]) and np.array_equal(tdX, gdX[sl]))
            res["tok_grad_err"] = max(float(np.abs(tsummed[(l, n)] - gg[l][n]).max() / (np.abs(gg[l][n]).max() + 1e-30))
                                      for l in range(cfg["L"]) for n in gg[l])
        q.put(res)
    finally:
        dist.destroy_process_group()


def test_two_rank_shards_match_full_batch():
    world = 2
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    res = [q.get(timeout=300) for _ in range(world)]
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    res = {r["rank"]: r for r in res}
    assert all(r["ok_mask"] for r in res.values())
    assert all(r["ms"] == 11.0 for r in res.values())  # slowest rank's time
    assert res[0]["out_ok"]
    assert res[0]["grad_err"] < 1e-12
    assert res[0]["tok_out_ok"]
    assert res[0]["tok_grad_err"] < 1e-12
