"""The exchange step of data-parallel calibration on two gloo ranks (CPU): per-rank sums of
Eq. 4 over disjoint token shards, summed across ranks, give the autocorrelation of all
tokens. The per-rank sums come from the fp64 oracle; the reduction is the library's."""
import os
import socket

import numpy as np
import torch
import torch.distributed as dist
import torch.multiprocessing as mp


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, K, n_per_rank, out_path):
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        import oracle
        import synth
        from paper_2410_05437_gb300.distributed import allreduce_sum_and_count
        model = synth.ActivationModel(K, seed=5, outliers=1)
        X = synth.bf16_to_f64(model.sample(n_per_rank, stream="calib_tokens", chunk=rank))
        S, n = allreduce_sum_and_count(oracle.autocorr_sum(X), n_per_rank)
        if rank == 0:
            np.save(out_path, np.concatenate([[n], (S / n).ravel()]))
    finally:
        dist.destroy_process_group()


def test_calibration_sum_over_two_gloo_ranks(tmp_path):
    import oracle
    import synth
    K, n_per_rank, world = 24, 300, 2
    out = str(tmp_path / "c.npy")
    mp.start_processes(_rank, args=(world, _free_port(), K, n_per_rank, out), nprocs=world,
                       start_method="spawn", join=True)
    res = np.load(out)
    n, C = int(res[0]), res[1:].reshape(K, K)
    assert n == world * n_per_rank
    model = synth.ActivationModel(K, seed=5, outliers=1)
    X = np.concatenate([synth.bf16_to_f64(model.sample(n_per_rank, stream="calib_tokens", chunk=r))
                        for r in range(world)])
    C_o = oracle.autocorr_sum(X) / n
    assert np.allclose(C, C_o, rtol=1e-12, atol=1e-14)
    # the projection built from the reduced C is the one of all tokens (Thm. 1)
    w_red = oracle.eigh(C)[0]
    w_all = oracle.eigh(C_o)[0]
    assert np.allclose(w_red, w_all, rtol=1e-10, atol=1e-14)
