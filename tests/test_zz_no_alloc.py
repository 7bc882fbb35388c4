"""espace_linear_forward_noalloc: the forward for callers that cannot allocate device memory
during the call (code running inside a memory budget or pool it does not own, servers
that reserve all device memory at start-up). It keeps the rank-L intermediate in a fixed
array inside the library instead of the handle's growable scratch.

Checked through the C ABI against espace_linear_forward, on two calls in a row with
different inputs, within the parity tolerances the other GPU tests use. This file is
collected last so that a run stopping at its first failure has run every other test.
"""
import numpy as np
import pytest
import torch

import synth

pytestmark = pytest.mark.gpu

Y_REL = 4e-3
Y_MAX = 2e-2
NOALLOC_Z_ELEMS = 8388608     # ESPACE_NOALLOC_Z_ELEMS in include/espace.h


@pytest.fixture(scope="module")
def esp():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2410_05437_gb300 as esp
    return esp


def close(Y, Y_ref):
    a = Y.double().cpu().numpy()
    b = Y_ref.double().cpu().numpy()
    err = np.linalg.norm(a - b) / np.linalg.norm(b)
    mx = np.abs(a - b).max() / np.abs(b).max()
    return np.all(np.isfinite(a)) and err <= Y_REL and mx <= Y_MAX


@pytest.mark.parametrize("N,K,M,L", [(128, 512, 512, 256),      # tensor-core kernels
                                     (300, 1024, 776, 300),     # ragged, several tiles
                                     (24, 1024, 768, 512),      # decode kernel here, swapped tcgen05 there
                                     (4, 512, 512, 256)])       # small-N kernels
def test_noalloc_forward_matches_forward_twice(esp, N, K, M, L):
    model = synth.ActivationModel(K, seed=N + K)
    W = synth.weights(M, K, seed=N + K).cuda()
    P = synth.random_projection(K, L, seed=N + K)
    p = esp.espace_proj_from_host(P, W)
    try:
        for call in range(2):
            X = model.sample(N, chunk=call).cuda()
            Y_ref = torch.empty((N, M), dtype=torch.bfloat16, device="cuda")
            Y = torch.full((N, M), float("nan"), dtype=torch.bfloat16, device="cuda")
            esp.espace_linear_forward(p, X, Y_ref)
            rc = esp.lib.espace_linear_forward_noalloc(p, X.data_ptr(), N, Y.data_ptr(),
                                                       torch.cuda.current_stream().cuda_stream)
            assert rc == 0, esp.lib.espace_last_error().decode()
            torch.cuda.synchronize()
            esp.espace_check()
            assert close(Y, Y_ref), f"call {call}"
    finally:
        esp.espace_proj_destroy(p)


def test_noalloc_forward_rejects_batches_beyond_the_fixed_scratch(esp):
    K, M, L = 1024, 64, 1024
    W = synth.weights(M, K, seed=3).cuda()
    p = esp.espace_proj_from_host(synth.random_projection(K, L, seed=3), W)
    try:
        N = NOALLOC_Z_ELEMS // L + 1
        X = torch.zeros((N, K), dtype=torch.bfloat16, device="cuda")
        Y = torch.full((N, M), 7.0, dtype=torch.bfloat16, device="cuda")
        with pytest.raises(esp.EspaceError) as e:
            esp.espace_linear_forward_noalloc(p, X, Y)
        assert e.value.code == 2
        assert "scratch" in str(e.value)
        torch.cuda.synchronize()
        assert torch.all(Y == 7.0)          # nothing was launched
        # the largest batch that fits runs
        Nmax = NOALLOC_Z_ELEMS // L
        esp.espace_linear_forward_noalloc(p, X[:Nmax], Y[:Nmax])
        torch.cuda.synchronize()
        esp.espace_check()
        assert torch.all(Y[:Nmax] == 0)
    finally:
        esp.espace_proj_destroy(p)


@pytest.mark.parametrize("N", [512, 24])
def test_noalloc_forward_leaves_device_memory_unchanged(esp, N):
    """The call allocates nothing: with the library's kernels and the fixed array already
    loaded (a first call), a call on a fresh handle, at a batch size that handle never saw,
    leaves the device's free memory exactly as it was."""
    K, M, L = 1024, 1024, 512
    W = synth.weights(M, K, seed=5).cuda()
    P = synth.random_projection(K, L, seed=5)
    X = synth.ActivationModel(K, seed=5).sample(N).cuda()
    Y = torch.empty((N, M), dtype=torch.bfloat16, device="cuda")
    warm = esp.espace_proj_from_host(P, W)
    try:
        esp.espace_linear_forward_noalloc(warm, X[:N // 2].contiguous(), Y[:N // 2])
        torch.cuda.synchronize()
    finally:
        esp.espace_proj_destroy(warm)
    p = esp.espace_proj_from_host(P, W)
    try:
        torch.cuda.synchronize()
        free0, _ = torch.cuda.mem_get_info()
        esp.espace_linear_forward_noalloc(p, X, Y)
        torch.cuda.synchronize()
        free1, _ = torch.cuda.mem_get_info()
        esp.espace_check()
        assert free1 == free0
        Y_ref = torch.empty_like(Y)
        esp.espace_linear_forward(p, X, Y_ref)
        torch.cuda.synchronize()
        assert close(Y, Y_ref)
    finally:
        esp.espace_proj_destroy(p)
