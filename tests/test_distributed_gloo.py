"""Host logic of the multi-rank step, on CPU with the gloo backend (world size 2).

Each rank takes its shard of the batch, computes the layer backward for it, and the
ranks sum the parameter gradients with one all-reduce. The result must equal the
backward of the whole batch on one process (the per-rank backward is the float64
oracle here: the CUDA kernels need a GPU, the exchange logic does not). With a
learnable somatic decay the exchanged buffer also carries dL/dbeta per channel.
"""
import os
import socket
import tempfile

import numpy as np
import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

from paper_2412_06355_gb300 import distributed, workloads

W = workloads.Workload("dp", T=5, B=5, N=2 * 48, K=4, G=1, C=2, inner=48, dtype="f32", psi="mh",
                       reset="hard", mask_p=0.7, seed=41)


def free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def rank_main(rank: int, world: int, port: int, out_dir: str, with_beta: bool):
    import oracle
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        inp = workloads.make_inputs(W, "cpu")
        b0, b1 = distributed.shard_range(W.B, world, rank)
        shard = W.with_(B=b1 - b0)
        sl = {k: v for k, v in inp.items()}
        sl["x"] = inp["x"][:, b0:b1].contiguous()
        sl["gs"] = inp["gs"][:, b0:b1].contiguous()
        g = oracle.backward_layer(shard, sl)
        flat, views = distributed.param_grad_buffer(W.C, W.K, W.Kb, with_beta=with_beta)
        for k in views:
            views[k].copy_(torch.from_numpy(g[k]).float())
        distributed.sum_param_grads(flat)
        np.save(os.path.join(out_dir, f"grads{rank}.npy"), flat.numpy())
        np.save(os.path.join(out_dir, f"gx{rank}.npy"), g["gx"])
    finally:
        dist.destroy_process_group()


def test_shard_range_covers_and_balances():
    for n in (0, 1, 5, 64, 129):
        for world in (1, 2, 3, 8):
            parts = [distributed.shard_range(n, world, r) for r in range(world)]
            assert parts[0][0] == 0 and parts[-1][1] == n
            assert all(parts[i][1] == parts[i + 1][0] for i in range(world - 1))
            sizes = [b - a for a, b in parts]
            assert max(sizes) - min(sizes) <= 1
    with pytest.raises(ValueError):
        distributed.shard_range(4, 2, 2)


def test_buffer_layout():
    C, K, Kb = 3, 4, 2
    for with_beta in (False, True):
        flat, views = distributed.param_grad_buffer(C, K, Kb, with_beta=with_beta)
        assert flat.numel() == 2 * C * K + 2 * C * Kb + (C if with_beta else 0)
        assert set(views) == {"galpha", "gxi", "gzeta", "gkappa"} | ({"gbeta"} if with_beta else set())
        flat.copy_(torch.arange(flat.numel(), dtype=torch.float32))
        row = distributed.split_param_grads(flat, C, K, Kb, with_beta)
        assert len(row) == (5 if with_beta else 4)
        assert torch.equal(torch.cat([r.reshape(-1) for r in row]), flat)   # views, in order
        assert row[2].shape == (C, Kb) and row[0].shape == (C, K)


@pytest.mark.parametrize("with_beta", [False, True], ids=["lif", "plif"])
def test_two_rank_gradient_sum_equals_whole_batch(with_beta):
    import oracle
    oracle.build()
    world = 2
    with tempfile.TemporaryDirectory() as d:
        mp.start_processes(rank_main, args=(world, free_port(), d, with_beta), nprocs=world,
                           start_method="spawn", join=True)
        summed = [np.load(os.path.join(d, f"grads{r}.npy")) for r in range(world)]
        gx = np.concatenate([np.load(os.path.join(d, f"gx{r}.npy")) for r in range(world)], axis=1)
    assert np.array_equal(summed[0], summed[1])            # every rank holds the same sum
    whole = oracle.backward_layer(W, workloads.make_inputs(W, "cpu"))
    flat, views = distributed.param_grad_buffer(W.C, W.K, W.Kb, with_beta=with_beta)
    for k in views:
        views[k].copy_(torch.from_numpy(whole[k]).float())
    np.testing.assert_allclose(summed[0], flat.numpy(), rtol=1e-5, atol=1e-6)
    if with_beta:                                          # dL/dbeta travels with the rest
        gb = distributed.split_param_grads(torch.from_numpy(summed[0]), W.C, W.K, W.Kb, True)[4]
        assert np.abs(whole["gbeta"]).max() > 0
        np.testing.assert_allclose(gb.numpy(), whole["gbeta"], rtol=1e-5, atol=1e-6)
    np.testing.assert_array_equal(gx, whole["gx"])           # neurons are independent
