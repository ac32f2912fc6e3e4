"""The N > 1 path on the CPU: two gloo ranks.

Windows are independent, so ranks shard them with no collective on the data path; only the
step time is reduced (max over ranks).  The reward's counter-based draws are keyed by the
global window index, so a sharded run reproduces the unsharded one exactly, and per-rank
loss partials (sum of w * E[L], |W|; with the anchor also sum KL and |positions|) combine
into the global loss with one all-reduce, for windows and for sharded sequences.  With the
data-parallel normalisers (the library's global_counts), one all-reduce of two integers before
the step gives |W| and |P| of the whole batch, and the ranks' losses normalised by them sum to
the whole batch's loss (the GPU side of that is tests/test_gpu_dp.py).
"""

import multiprocessing as mp
import os
import socket

import numpy as np
import pytest
import torch


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    import torch.distributed as dist
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        import bench
        import oracle
        import synth
        res = {"max": bench.max_over_ranks(float(10 * (rank + 1)), world)}
        # the whole batch, drawn identically on every rank; each rank keeps its shard
        target, draft, _ = synth.make_logits("tiny", seed=3, N=8, K=4, V=64)
        per = 8 // world
        lo = bench.rank_row_offset(rank, per)
        t, d = target[lo:lo + per], draft[lo:lo + per]
        rw = oracle.accept_reward(t, d, None, 2, 0.9, seed=7, row_offset=lo, windows_per_rollout=2,
                                  rollouts_per_group=2)
        taus = [torch.zeros(per, dtype=torch.int64) for _ in range(world)]
        dist.all_gather(taus, torch.as_tensor(rw["tau"]))
        res["tau"] = torch.cat(taus).numpy()
        fw = oracle.loss_forward(t, d, None, oracle.MODE_BOTH, 0.9, 0.5, 0.5)
        part = torch.tensor([0.5 * fw["eal_g"].sum() + 0.5 * fw["eal_s"].sum(), float(fw["nvalid"])],
                            dtype=torch.float64)
        dist.all_reduce(part)
        res["loss"] = float(-part[0] / part[1])
        # sequence layout, sequences sharded: the partials of L_KL + 0.1 L_EAL are
        # (sum E^g, |W|, sum KL, |positions|), one all-reduce of four numbers
        st, sd, sm = synth.make_seq_logits("seq_tiny", seed=4, B=4, seq_len=11, V=50)
        bper = 4 // world
        b0 = rank * bper
        ts, ds, ms = st[b0:b0 + bper], sd[b0:b0 + bper], sm[b0:b0 + bper].numpy()
        fe = oracle.seq_loss_forward(ts, ds, ms, 3, oracle.MODE_GREEDY)
        an = oracle.anchor_forward(ts, ds, ms)
        sp = torch.tensor([fe["eal_g"].sum(), float(fe["nvalid"]), float(np.sum(an["kl"][an["valid"]])),
                           float(an["npos"])], dtype=torch.float64)
        dist.all_reduce(sp)
        res["seq_loss"] = float(-0.1 * sp[0] / sp[1] + sp[2] / sp[3])
        # data-parallel normalisers (the library's global_counts): each rank counts its shard's |W|
        # (windows whose depth 0 is valid) and |P| (valid positions), one all-reduce of the two
        # integers gives the whole batch's, and each rank's objective normalised by them; the
        # ranks' losses then sum to the whole batch's, with no collective on the data path
        tg, dg, mg = synth.make_logits("tiny", seed=5, N=8, K=4, V=64, mask_rate=0.3)
        ml = mg[lo:lo + per].numpy()
        counts = torch.tensor([int((ml[:, 0] != 0).sum()), int((ml != 0).sum())], dtype=torch.int64)
        dist.all_reduce(counts)
        nW, nP = int(counts[0]), int(counts[1])
        omode = oracle.MODE_KL | oracle.MODE_BOTH
        lr = oracle.objective_forward(tg[lo:lo + per], dg[lo:lo + per], ml, omode, 0.9, 0.5, 0.5, 1.0, nW, nP)["loss"]
        tot = torch.tensor([lr], dtype=torch.float64)
        dist.all_reduce(tot)
        res["dp_counts"] = (nW, nP)
        res["dp_loss"] = float(tot[0])
        out.put((rank, res))
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks():
    ctx = mp.get_context("spawn")
    out = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, out)) for r in range(2)]
    for p in procs:
        p.start()
    results = dict(out.get(timeout=240) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    import oracle
    import synth
    target, draft, _ = synth.make_logits("tiny", seed=3, N=8, K=4, V=64)
    whole = oracle.accept_reward(target, draft, None, 2, 0.9, seed=7, row_offset=0, windows_per_rollout=2,
                                 rollouts_per_group=2)
    ref_loss = oracle.loss_forward(target, draft, None, oracle.MODE_BOTH, 0.9, 0.5, 0.5)["loss"]
    st, sd, sm = synth.make_seq_logits("seq_tiny", seed=4, B=4, seq_len=11, V=50)
    ref_seq = oracle.seq_objective_forward(st, sd, sm.numpy(), 3, oracle.MODE_KL | oracle.MODE_GREEDY, 1.0,
                                           0.1, 0.0, 1.0)["loss"]
    tg, dg, mg = synth.make_logits("tiny", seed=5, N=8, K=4, V=64, mask_rate=0.3)
    mh = mg.numpy()
    ref_dp = oracle.objective_forward(tg, dg, mh, oracle.MODE_KL | oracle.MODE_BOTH, 0.9, 0.5, 0.5, 1.0)["loss"]
    for r in range(2):
        assert results[r]["dp_counts"] == (int((mh[:, 0] != 0).sum()), int((mh != 0).sum()))
        assert abs(results[r]["dp_loss"] - ref_dp) < 1e-12
        assert results[r]["max"] == 20.0
        np.testing.assert_array_equal(results[r]["tau"], whole["tau"])
        assert abs(results[r]["loss"] - ref_loss) < 1e-12
        assert abs(results[r]["seq_loss"] - ref_seq) < 1e-12
