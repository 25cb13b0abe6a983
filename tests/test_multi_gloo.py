"""Multi-process host logic on CPU with the gloo backend, world size 2: sequence sharding of one
evaluation (size-weighted all-reduce equals the full batch, computed here with the oracle on each
shard, for the MSE term and for the joint MSE + KL objective), the Fisher-coupling score of a
sharded evaluation (norm of the combined weight gradient), and the max-over-ranks timing reduction
used by bench.py."""
import os
import socket

import numpy as np
import pytest
import torch
import torch.multiprocessing as mp


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _worker(rank, world, port, out):
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        from oracle import jab_oracle as O
        from paper_2609_34866_gb300.multi import (combine_shards, dist_env,
                                                  fisher_score_from_shards, max_over_ranks,
                                                  shard_sequences)
        assert dist_env() == (world, rank, rank)
        rng = np.random.default_rng(0)
        B, T, d = 5, 6, 8
        desc = dict(d_model=d, n_q_heads=2, n_kv_heads=1, head_dim=4, group_size=4, use_rope=True,
                    rope_theta=10000.0, softmax_scale=0.0)
        x = rng.standard_normal((B, T, d))
        w = rng.standard_normal((16, d)) * 0.3
        s = O.init_scales_absmax(w, 3, 4)
        a, b = shard_sequences(B, world, rank)
        r = O.jab_loss_and_grad(x[a:b], w, s, 3, desc, kappa=1.0)
        loss = torch.tensor([r["loss"]], dtype=torch.float64)
        grad = torch.tensor(r["grad_s"], dtype=torch.float64)
        combine_shards(loss, grad, b - a, B)
        gw = torch.tensor(r["grad_w_hat"], dtype=torch.float64)
        score = fisher_score_from_shards(gw, b - a, B)
        # the joint objective (MSE + 0.1 KL, Eq. 3): the KL batchmean shards like the MSE mean
        rj = O.jab_loss_joint_and_grad(x[a:b], w, s, 3, desc, lam_kl=0.1, kappa=1.0)
        jloss = torch.tensor([rj["loss"]], dtype=torch.float64)
        jgrad = torch.tensor(rj["grad_s"], dtype=torch.float64)
        combine_shards(jloss, jgrad, b - a, B)
        t = max_over_ranks(10.0 + rank)
        if rank == 0:
            jfull = O.jab_loss_joint_and_grad(x, w, s, 3, desc, lam_kl=0.1, kappa=1.0)
            out["jloss"] = (jloss.item(), jfull["loss"])
            out["jgrad"] = float(np.abs(jgrad.numpy() - jfull["grad_s"]).max() /
                                 np.abs(jfull["grad_s"]).max())
            full = O.jab_loss_and_grad(x, w, s, 3, desc, kappa=1.0)
            out["loss"] = (loss.item(), full["loss"])
            out["grad"] = float(np.abs(grad.numpy() - full["grad_s"]).max() /
                                np.abs(full["grad_s"]).max())
            out["tmax"] = t
            out["score"] = (score, float((full["grad_w_hat"] ** 2).sum()))
    finally:
        dist.destroy_process_group()


def test_shard_ranges_cover_the_batch():
    from paper_2609_34866_gb300.multi import shard_sequences
    for B in (1, 2, 5, 128):
        for world in (1, 2, 3, 8):
            ranges = [shard_sequences(B, world, r) for r in range(world)]
            assert ranges[0][0] == 0 and ranges[-1][1] == B
            assert all(r1[1] == r2[0] for r1, r2 in zip(ranges, ranges[1:]))
            assert max(b - a for a, b in ranges) - min(b - a for a, b in ranges) <= 1


def test_sharded_evaluation_matches_full_batch_gloo_world2():
    ctx = mp.get_context("spawn")
    with ctx.Manager() as mgr:
        out = mgr.dict()
        mp.start_processes(_worker, args=(2, _free_port(), out), nprocs=2, join=True,
                           start_method="spawn")
        loss_sharded, loss_full = out["loss"]
        np.testing.assert_allclose(loss_sharded, loss_full, rtol=1e-12)
        assert out["grad"] < 1e-12
        assert out["tmax"] == 11.0
        score_sharded, score_full = out["score"]
        np.testing.assert_allclose(score_sharded, score_full, rtol=1e-12)
        jl_sharded, jl_full = out["jloss"]
        np.testing.assert_allclose(jl_sharded, jl_full, rtol=1e-12)
        assert out["jgrad"] < 1e-12
