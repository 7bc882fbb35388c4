"""Data-parallel calibration end to end over two processes (Eq. 4; the one exchange step of
the data-parallel path): each rank accumulates its own token shard on the GPU, the sums and
counts are added across ranks on the host (gloo) by distributed.calib_allreduce (export,
fp64 all-reduce, import), and every rank then builds the projection (Thm. 1) from the
reduced sum. Both processes share the one GPU; no kernel of one waits on the other's.

Checked against the oracle over the union of the shards: C = S / n, the count, the
eigenvalues and the L-dimensional subspace (Davis-Kahan bound), and both ranks' projections
agree bit for bit."""
import os
import socket

import numpy as np
import pytest
import torch
import torch.multiprocessing as mp

import synth

pytestmark = pytest.mark.gpu

K, M, L, N_PER_RANK, WORLD = 256, 192, 64, 1536, 2


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, out_dir):
    import torch.distributed as dist
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        torch.cuda.set_device(0)
        import paper_2410_05437_gb300 as esp
        from paper_2410_05437_gb300.distributed import calib_allreduce
        model = synth.ActivationModel(K, seed=17)
        X = model.sample(N_PER_RANK, stream="calib_tokens", chunk=rank).cuda()
        W = synth.weights(M, K, seed=17).cuda()
        h = esp.espace_calib_create(K)
        p = None
        try:
            # two accumulate calls per rank, as a rank would over its local batches
            esp.espace_calib_accumulate(h, X[: N_PER_RANK // 3].contiguous())
            esp.espace_calib_accumulate(h, X[N_PER_RANK // 3:].contiguous())
            n = calib_allreduce(h, K)
            C, cnt = esp.espace_calib_read(h, K)
            p = esp.espace_build_projection(h, W, L)
            w = esp.espace_proj_eigenvalues(p)
            P_bits = esp.espace_proj_read_P(p)
            esp.espace_check()
            np.savez(os.path.join(out_dir, f"rank{rank}.npz"), C=C, n=np.array([n, cnt]), w=w, P=P_bits)
        finally:
            if p:
                esp.espace_proj_destroy(p)
            esp.espace_calib_destroy(h)
    finally:
        dist.destroy_process_group()


def test_calibration_allreduce_two_processes_build_projection(tmp_path):
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import oracle
    mp.start_processes(_rank, args=(WORLD, _free_port(), str(tmp_path)), nprocs=WORLD,
                       start_method="spawn", join=True)
    res = [np.load(os.path.join(tmp_path, f"rank{r}.npz")) for r in range(WORLD)]
    model = synth.ActivationModel(K, seed=17)
    X = np.concatenate([synth.bf16_to_f64(model.sample(N_PER_RANK, stream="calib_tokens", chunk=r))
                        for r in range(WORLD)])
    n = WORLD * N_PER_RANK
    S_o = oracle.autocorr_sum(X)
    C_o = S_o / n
    P_o, _, w_o, _ = oracle.build_projection(S_o, n, L)
    for r in res:
        assert list(r["n"]) == [n, n]
        err = np.linalg.norm(r["C"] - C_o) / np.linalg.norm(C_o)
        assert err <= 1e-5, f"C normwise {err:.3e}"
        assert np.allclose(r["w"], w_o, rtol=0, atol=1e-5 * w_o[0])
        Pb = synth.bf16_to_f64(torch.from_numpy(r["P"].view(np.int16)).view(torch.bfloat16))
        gap = w_o[L - 1] - w_o[L]
        proj = np.linalg.norm(Pb @ Pb.T - P_o @ P_o.T, 2)
        assert proj <= 1e-5 * np.linalg.norm(C_o) / gap + 2e-2, proj
    # both ranks hold the same reduced sum, so they build the same projection
    assert np.array_equal(res[0]["C"], res[1]["C"])
    assert np.array_equal(res[0]["P"], res[1]["P"])
