"""Data-parallel contract of the loss head, checked with two gloo ranks on CPU:
sharding by trajectory plus one all-reduced action-token count (n_norm) makes
the sum of the per-rank policy and value losses and of the weight gradients
equal the unsplit batch, and the value gradients its slices.
The arithmetic on each rank is the fp64 oracle (no GPU here)."""
import os
import socket

import numpy as np
import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

from paper_2607_07508_gb300 import dp, synthetic as S


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out):
    from oracle import sao_oracle as O
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        wl = S.make_custom([40, 7, 0, 63, 25, 90, 3], 16, 50, "f32", seed=42, obs_frac=0.3)
        arrays = {"values_tok": wl.values, "mask_tok": wl.loss_mask, "y_tok": wl.y, "xi_tok": wl.xi,
                  "H_tok": wl.H.numpy(), "rewards_traj": wl.rewards}
        shard = dp.shard_trajectories(wl.cu_seqlens, world)[rank]
        loc, cu = dp.local_batch(arrays, wl.cu_seqlens, shard)
        adv, _ = O.advantages(loc["values_tok"], loc["rewards_traj"], loc["mask_tok"], cu, 1.0, 0.95, 1.0)
        logp, lse = O.token_logprobs(loc["H_tok"], wl.W, loc["y_tok"])
        old = logp + loc["xi_tok"]
        n_norm = dp.global_action_count(int(loc["mask_tok"].sum()))
        pl = O.policy_loss(logp, old, adv, loc["mask_tok"], 0.2, 0.28, n_norm=n_norm)
        _, dW = O.token_logprobs_bwd(loc["H_tok"], wl.W, loc["y_tok"], lse, pl["coef"])
        ret_loc = loc["values_tok"] + 0.5 * loc["xi_tok"]
        vl, vg, _ = O.value_loss(loc["values_tok"], ret_loc, loc["mask_tok"], n_norm=n_norm)
        t_loss = torch.tensor([pl["loss"]], dtype=torch.float64)
        t_vloss = torch.tensor([vl], dtype=torch.float64)
        t_dW = torch.tensor(dW)
        dist.all_reduce(t_loss)
        dist.all_reduce(t_vloss)
        dist.all_reduce(t_dW)
        # each rank's value gradient is its slice of the unsplit batch's
        t0, t1 = int(wl.cu_seqlens[shard[0]]), int(wl.cu_seqlens[shard[1]])
        _, vg_f, _ = O.value_loss(wl.values, wl.values + 0.5 * wl.xi, wl.loss_mask)
        out[f"vgrad{rank}"] = float(np.abs(vg - vg_f[t0:t1]).max())
        if rank == 0:
            adv_f, _ = O.advantages(wl.values, wl.rewards, wl.loss_mask, wl.cu_seqlens, 1.0, 0.95, 1.0)
            lp_f, lse_f = O.token_logprobs(wl.H, wl.W, wl.y)
            pl_f = O.policy_loss(lp_f, lp_f + wl.xi, adv_f, wl.loss_mask, 0.2, 0.28)
            _, dW_f = O.token_logprobs_bwd(wl.H, wl.W, wl.y, lse_f, pl_f["coef"])
            out["loss"] = (float(t_loss.item()), pl_f["loss"])
            out["vloss"] = (float(t_vloss.item()), O.value_loss(wl.values, wl.values + 0.5 * wl.xi, wl.loss_mask)[0])
            out["dW"] = float(np.abs(t_dW.numpy() - dW_f).max()), float(np.abs(dW_f).max())
            out["n_norm"] = (n_norm, int(wl.loss_mask.sum()))
    finally:
        dist.destroy_process_group()


def test_shard_covers_every_trajectory_once():
    cu = np.array([0, 5, 5, 9, 30, 31, 60])
    for world in (1, 2, 3, 4, 8):
        shards = dp.shard_trajectories(cu, world)
        assert shards[0][0] == 0 and shards[-1][1] == len(cu) - 1
        for (a0, a1), (b0, b1) in zip(shards, shards[1:]):
            assert a1 == b0 and a0 <= a1


def test_two_gloo_ranks_match_unsplit_batch():
    ctx = mp.get_context("spawn")
    mgr = ctx.Manager()
    out = mgr.dict()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, 2, port, out)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=240)
    assert all(p.exitcode == 0 for p in procs), [p.exitcode for p in procs]
    got, want = out["loss"]
    assert abs(got - want) <= 1e-12 * max(1.0, abs(want))
    err, scale = out["dW"]
    assert err <= 1e-12 * max(1.0, scale)
    assert out["n_norm"][0] == out["n_norm"][1]
    got, want = out["vloss"]
    assert abs(got - want) <= 1e-12 * max(1.0, abs(want))
    assert out["vgrad0"] <= 1e-15 and out["vgrad1"] <= 1e-15
