"""Parity of the CUDA path (through the C ABI) with the fp64 oracle, on the same seeded inputs.

Tolerances: on Y, normwise ||Y - Y_o||_F / ||Y_o||_F <= 4e-3 and max |Y - Y_o| <= 2e-2 max |Y_o|;
on C = S / n, normwise 1e-5. Z is rounded to bf16 on both sides (fp32 accumulation on the
GPU, fp64 in the oracle), so isolated one-ulp flips of Z at rounding ties are expected and
covered by the Y tolerance.
"""
import time

import numpy as np
import pytest
import torch

import oracle
import synth

pytestmark = pytest.mark.gpu

Y_REL = 4e-3
Y_MAX = 2e-2
C_REL = 1e-5


@pytest.fixture(scope="module")
def esp():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2410_05437_gb300 as esp
    return esp


def dev(t):
    return t.to("cuda").contiguous()


def f64(t):
    return synth.bf16_to_f64(t.cpu())


def assert_y_close(Y_gpu, Y_ref):
    Y = f64(Y_gpu) if isinstance(Y_gpu, torch.Tensor) else Y_gpu
    err = np.linalg.norm(Y - Y_ref) / max(np.linalg.norm(Y_ref), 1e-300)
    mx = np.abs(Y - Y_ref).max() / max(np.abs(Y_ref).max(), 1e-300)
    assert np.all(np.isfinite(Y))
    assert err <= Y_REL, f"normwise error {err:.3e}"
    assert mx <= Y_MAX, f"max error {mx:.3e}"
    return err, mx


def make_layer(K, M, N, seed, outliers=None, sigma=0.5):
    model = synth.ActivationModel(K, seed=seed, outliers=outliers, lognormal_sigma=sigma)
    X = model.sample(N)
    W = synth.weights(M, K, seed=seed)
    return model, X, W


# ------------------------------------------------------------------------------ dense (Eq. 1)

@pytest.mark.parametrize("N,K,M", [(128, 512, 512), (200, 520, 264), (1, 64, 8), (300, 1024, 776),
                                   (129, 136, 392), (9, 136, 392), (32, 520, 264), (5, 4096, 12288),
                                   (33, 2056, 1000), (256, 1024, 776), (512, 4096, 2056), (300, 8192, 776), (128, 4096, 12288)])
def test_dense_forward_matches_oracle(esp, N, K, M):
    _, X, W = make_layer(K, M, N, seed=100 + N)
    Y = torch.empty((N, M), dtype=torch.bfloat16, device="cuda")
    esp.espace_dense_forward(dev(X), dev(W), Y)
    torch.cuda.synchronize()
    assert_y_close(Y, oracle.dense(f64(X), f64(W)))
    esp.espace_check()


# ------------------------------------------------------------------------------ fold and P

def test_projection_upload_and_fold(esp):
    K, M, L = 512, 512, 256
    P = synth.random_projection(K, L, seed=7)
    W = synth.weights(M, K, seed=7)
    p = esp.espace_proj_from_host(P, dev(W))
    try:
        Pb = esp.espace_proj_read_P(p)
        want = oracle.bf16_round(P)
        assert np.array_equal(Pb.view(np.uint16), synth.bf16_bits(torch.from_numpy(want).to(torch.bfloat16)))
        Wf = synth.bf16_to_f64(torch.from_numpy(esp.espace_proj_read_Wfold(p).view(np.int16)).view(torch.bfloat16))
        Wf_o = oracle.fold(want, f64(W))
        # fp32 (GPU) vs fp64 (oracle) accumulation: the fp32 sum is within
        # K * 2^-24 * sum_k |P[k][l] W[m][k]| of the exact one, then both round to bf16
        # (one ulp each way at most); most entries agree exactly
        acc_bound = K * 2.0 ** -24 * oracle.fold(np.abs(want), np.abs(f64(W)), round_bf16=False)
        ulp = np.abs(Wf_o) * 2.0 ** -7
        diff = np.abs(Wf - Wf_o)
        assert np.all(diff <= ulp + 2 * acc_bound)
        assert np.mean(diff > 0) < 0.02
    finally:
        esp.espace_proj_destroy(p)


def test_projection_from_device_matches_host_path(esp):
    """A bf16 P^T handed over on the device gives the same handle as the fp64 host path
    after its rounding: bit-identical P and W', and the same outputs."""
    K, M, L, N = 520, 264, 100, 40
    P = synth.random_projection(K, L, seed=11)
    W = dev(synth.weights(M, K, seed=11))
    Pb = oracle.bf16_round(P)
    PT = torch.from_numpy(np.ascontiguousarray(Pb.T)).to(torch.bfloat16).cuda()
    a = esp.espace_proj_from_host(P, W)
    b = esp.espace_proj_from_device(PT, W)
    try:
        assert np.array_equal(esp.espace_proj_read_P(a), esp.espace_proj_read_P(b))
        assert np.array_equal(esp.espace_proj_read_Wfold(a), esp.espace_proj_read_Wfold(b))
        _, X, _ = make_layer(K, M, N, seed=11)
        Ya = torch.empty((N, M), dtype=torch.bfloat16, device="cuda")
        Yb = torch.empty_like(Ya)
        esp.espace_linear_forward(a, dev(X), Ya)
        esp.espace_linear_forward(b, dev(X), Yb)
        torch.cuda.synchronize()
        esp.espace_check()
        assert torch.equal(Ya.view(torch.int16), Yb.view(torch.int16))
    finally:
        esp.espace_proj_destroy(a)
        esp.espace_proj_destroy(b)


# ------------------------------------------------------------------------------ forward (Eq. 3)

FORWARD_CASES = [
    # (N, K, M, L, path)
    (128, 512, 512, 256, 1),       # the tiny configuration
    (200, 520, 264, 100, 1),       # ragged N, K, M and L (padded to 128)
    (257, 1024, 3000, 300, 1),     # several tiles and a ragged tail
    (1, 512, 512, 256, 2),
    (3, 520, 264, 100, 2),
    (8, 1024, 776, 448, 2),
    (8, 1024, 776, 448, 1),        # the same shape on both kernel families
    (5, 512, 512, 512, 0),         # full rank, automatic path
    (17, 520, 264, 100, 2),        # decode kernel with 16- and 32-token groups, ragged
    (32, 1024, 776, 448, 2),
    (12, 512, 4104, 256, 2),       # M not a multiple of the 32-row tile
    (32, 1024, 776, 448, 1),
    (600, 1024, 1000, 512, 1),     # one persistent launch for both products, ragged M
    (600, 1024, 1000, 512, 3),     # the same on two launches
    (1000, 2048, 2312, 1000, 1),   # fused, ragged N / L / M, several row blocks
    (777, 2048, 1000, 256, 0),     # K >= 2 M and few Z tiles: rank-L product split over the SMs
    (300, 1040, 264, 64, 1),       # the same just above the swapped token range, ragged K
    (2304, 1152, 520, 1152, 1),    # 45 Z tiles: one persistent launch for both products
    (512, 4096, 12288, 2048, 1),   # fused, more Y tiles than CTA pairs
    (700, 6144, 1000, 520, 1),     # K >= 2 M: rank-L product split over the SMs, ragged N / L / M
    (300, 1024, 3000, 300, 3),
    # few tokens on tcgen05 with the weights as the 128-row operand; split reductions
    (100, 4096, 776, 2048, 1),     # both products split (16 and 7 weight tiles)
    (33, 1040, 3000, 600, 0),      # ragged N, K (not a multiple of 64), L and M
    (256, 2048, 1000, 1000, 0),    # 256-token tiles
    (129, 520, 264, 100, 1),       # 256-token tile, ragged
    (7, 1024, 776, 448, 1),        # fewer tokens than one MMA's rows
    (128, 4096, 12288, 2048, 0),   # Llama2 QKV at 128 tokens
    # one token on the decode kernel, across its stage layouts
    (1, 4096, 12288, 2048, 0),     # Llama2 QKV layer
    (1, 11008, 4096, 1376, 2),     # K beyond one 2048-wide k-block, ragged
    (1, 1040, 22016, 600, 0),      # wide M, ragged L, K not a multiple of 64
    (1, 24, 8, 1, 0),              # rank 1
    (1, 16384, 264, 128, 0),       # large K, few output rows
    (1, 24576, 512, 128, 2),       # K of the GPT3-22B FC2 layer
    # phase 2 over several 2048-wide k-blocks of Z, the last one ragged
    (4, 8192, 520, 4500, 2),       # three k-blocks, ragged M tail
    (32, 4096, 776, 3000, 2),      # two k-blocks, 32-token groups
]


def test_launch_counts(esp):
    K, M, L = 1024, 1000, 512
    P = synth.random_projection(K, L, seed=2)
    p = esp.espace_proj_from_host(P, dev(synth.weights(M, K, seed=2)))
    try:
        assert esp.espace_linear_forward_launches(p, 0) == 0
        assert esp.espace_linear_forward_launches(p, 1) == 1          # decode kernel
        assert esp.espace_linear_forward_launches(p, 600) == 1        # fused
        assert esp.espace_linear_forward_launches(p, 600, esp.PATH_TENSOR_SPLIT) == 2
        # few tokens: both products split their reduction here (4 and 8 weight tiles), each
        # followed by the launch that adds the partials
        assert esp.espace_linear_forward_launches(p, 100, esp.PATH_TENSOR) == 4
        assert esp.espace_linear_forward_launches(p, 64, esp.PATH_SMALL_N) == -1
    finally:
        esp.espace_proj_destroy(p)
    # K >= 2 M with 12 Z tiles at 600 tokens: the rank-L product splits its reduction (one
    # launch for the partials, one adding them), then the folded-weight product
    K, M, L = 2048, 1000, 512
    p = esp.espace_proj_from_host(synth.random_projection(K, L, seed=3), dev(synth.weights(M, K, seed=3)))
    try:
        assert esp.espace_linear_forward_launches(p, 600) == 3
        assert esp.espace_linear_forward_launches(p, 600, esp.PATH_TENSOR_SPLIT) == 3
        assert esp.espace_linear_forward_launches(p, 4864) == 1      # 38 Z tiles: fused
    finally:
        esp.espace_proj_destroy(p)


@pytest.mark.parametrize("N,K,M,L,path", FORWARD_CASES)
def test_linear_forward_matches_oracle(esp, N, K, M, L, path):
    seed = 1000 + N + K + L
    _, X, W = make_layer(K, M, N, seed=seed)
    P = synth.random_projection(K, L, seed=seed)
    p = esp.espace_proj_from_host(P, dev(W))
    try:
        Y = torch.full((N, M), float("nan"), dtype=torch.bfloat16, device="cuda")
        esp.espace_linear_forward_path(p, dev(X), Y, path)
        torch.cuda.synchronize()
        esp.espace_check()
        Y_o, _, _ = oracle.forward(f64(X), oracle.bf16_round(P), f64(W))
        assert_y_close(Y, Y_o)
    finally:
        esp.espace_proj_destroy(p)


def test_few_token_forward_is_reproducible(esp):
    """The split reductions add their fp32 partials in a fixed order: two calls give the
    same bits."""
    N, K, M, L = 96, 4096, 1000, 2048
    _, X, W = make_layer(K, M, N, seed=31)
    P = synth.random_projection(K, L, seed=31)
    p = esp.espace_proj_from_host(P, dev(W))
    try:
        Xd = dev(X)
        Y1 = torch.empty((N, M), dtype=torch.bfloat16, device="cuda")
        Y2 = torch.empty_like(Y1)
        esp.espace_linear_forward(p, Xd, Y1)
        esp.espace_linear_forward(p, Xd, Y2)
        torch.cuda.synchronize()
        esp.espace_check()
        assert torch.equal(Y1.view(torch.int16), Y2.view(torch.int16))
        Y_o, _, _ = oracle.forward(f64(X), oracle.bf16_round(P), f64(W))
        assert_y_close(Y1, Y_o)
    finally:
        esp.espace_proj_destroy(p)


@pytest.mark.parametrize("N", [1, 700, 2304, 4100])
def test_linear_forward_host_buffers(esp, N):
    """X and Y in pinned host memory: chunks of the tokens copied in, computed and copied
    out on overlapping streams; the result matches the device-buffer forward and the oracle."""
    K, M, L = 1024, 1000, 512
    _, X, W = make_layer(K, M, N, seed=6000 + N)
    P = synth.random_projection(K, L, seed=6000 + N)
    p = esp.espace_proj_from_host(P, dev(W))
    try:
        Xh = X.contiguous().pin_memory()
        Yh = torch.full((N, M), float("nan"), dtype=torch.bfloat16).pin_memory()
        esp.espace_linear_forward_host(p, Xh, Yh)
        esp.espace_check()
        assert_y_close(Yh, oracle.forward(f64(X), oracle.bf16_round(P), f64(W))[0])
        Yd = torch.empty((N, M), dtype=torch.bfloat16, device="cuda")
        esp.espace_linear_forward(p, dev(X), Yd)
        torch.cuda.synchronize()
        if N >= 1024:   # the same fused kernel on chunks of more than 256 tokens
            assert torch.equal(Yh.view(torch.int16), Yd.cpu().view(torch.int16))
    finally:
        esp.espace_proj_destroy(p)


def test_linear_forward_host_async_two_layers_on_two_streams(esp):
    """The asynchronous host-buffer forward: two layers, each on a stream of its own, two
    calls each with different inputs queued back to back (the second call on a handle reuses
    its staging, so it must run after the first), nothing waited for until both streams are
    synchronized; every output equals the device-buffer forward bit for bit, and the oracle
    within the tolerances."""
    # K < 2 M: the fused kernel; 16,500 tokens: two chunks (8448 + 8052), 1300: one
    shapes = [(1024, 1000, 512, 16500), (1536, 1000, 448, 1300)]
    layers = []
    try:
        for i, (K, M, L, N) in enumerate(shapes):
            model = synth.ActivationModel(K, seed=6100 + i)
            W = synth.weights(M, K, seed=6100 + i)
            P = synth.random_projection(K, L, seed=6100 + i)
            p = esp.espace_proj_from_host(P, dev(W))
            Xs = [model.sample(N, chunk=c).contiguous().pin_memory() for c in range(2)]
            Ys = [torch.full((N, M), float("nan"), dtype=torch.bfloat16).pin_memory() for _ in range(2)]
            layers.append({"p": p, "P": P, "W": W, "X": Xs, "Y": Ys, "s": torch.cuda.Stream()})
        torch.cuda.synchronize()
        for c in range(2):
            for l in layers:
                esp.espace_linear_forward_host_async(l["p"], l["X"][c], l["Y"][c], l["s"])
        for l in layers:
            l["s"].synchronize()
        esp.espace_check()
        for l in layers:
            for c in range(2):
                N, M = l["Y"][c].shape
                Yd = torch.empty((N, M), dtype=torch.bfloat16, device="cuda")
                esp.espace_linear_forward(l["p"], dev(l["X"][c]), Yd)
                torch.cuda.synchronize()
                assert torch.equal(l["Y"][c].view(torch.int16), Yd.cpu().view(torch.int16))
                Y_o = oracle.forward(f64(l["X"][c]), oracle.bf16_round(l["P"]), f64(l["W"]))[0]
                assert_y_close(l["Y"][c], Y_o)
    finally:
        for l in layers:
            esp.espace_proj_destroy(l["p"])


def test_linear_forward_host_many_layers_in_one_pipeline(esp):
    """Several independent layers through one host-buffer pipeline: one copy-in stream, the
    products in layer order on the caller's stream, one copy-out stream. Every output equals
    the device-buffer forward bit for bit (chunks of at least 2048 tokens all run the fused
    kernel, whose per-token sums do not depend on the batch) and the oracle within the
    tolerances. A layer with N = 0 is skipped, an empty list is a no-op, and a repeated
    handle or more than 16 layers is refused before anything is queued."""
    # 16,500 tokens, the first layer: chunks of 2048, 4096, 5376 and 4980 tokens; 300 and 1
    # token: one chunk each (the fused launch, the decode kernel)
    shapes = [(1024, 1000, 512, 16500), (1536, 776, 448, 300), (512, 520, 256, 0), (1040, 264, 100, 1)]
    layers = []
    try:
        for i, (K, M, L, N) in enumerate(shapes):
            model = synth.ActivationModel(K, seed=6200 + i)
            W = synth.weights(M, K, seed=6200 + i)
            P = synth.random_projection(K, L, seed=6200 + i)
            p = esp.espace_proj_from_host(P, dev(W))
            X = model.sample(N).contiguous().pin_memory() if N > 0 else torch.empty((0, K), dtype=torch.bfloat16)
            Y = torch.full((max(N, 1), M), float("nan"), dtype=torch.bfloat16).pin_memory()[:N]
            layers.append({"p": p, "P": P, "W": W, "X": X, "Y": Y})
        for rep in range(2):   # the second call reuses every handle's staging
            for l in layers:
                l["Y"].fill_(float("nan"))
            esp.espace_linear_forward_host_many([l["p"] for l in layers], [l["X"] for l in layers],
                                                [l["Y"] for l in layers])
            esp.espace_check()
            for l in layers:
                N, M = l["Y"].shape
                if N == 0:
                    continue
                Yd = torch.empty((N, M), dtype=torch.bfloat16, device="cuda")
                esp.espace_linear_forward(l["p"], dev(l["X"]), Yd)
                torch.cuda.synchronize()
                assert torch.equal(l["Y"].view(torch.int16), Yd.cpu().view(torch.int16))
                if rep == 0:
                    Y_o = oracle.forward(f64(l["X"]), oracle.bf16_round(l["P"]), f64(l["W"]))[0]
                    assert_y_close(l["Y"], Y_o)
        esp.espace_linear_forward_host_many([], [], [])
        with pytest.raises(esp.EspaceError) as e:
            esp.espace_linear_forward_host_many([layers[0]["p"], layers[0]["p"]], [layers[0]["X"]] * 2,
                                                [layers[0]["Y"]] * 2)
        assert e.value.code == 1                        # ESPACE_ERR_ARG
        with pytest.raises(esp.EspaceError) as e:
            esp.espace_linear_forward_host_many([layers[3]["p"]] * 17, [layers[3]["X"]] * 17, [layers[3]["Y"]] * 17)
        assert e.value.code == 1                        # ESPACE_ERR_ARG
    finally:
        for l in layers:
            esp.espace_proj_destroy(l["p"])


def test_linear_forward_full_rank_equals_dense_within_bf16(esp):
    """L = K: P P^T = I, so the projected layer reproduces the dense one (Sec. 2.2)."""
    N, K, M = 64, 256, 384
    _, X, W = make_layer(K, M, N, seed=77)
    P = synth.random_projection(K, K, seed=77)
    p = esp.espace_proj_from_host(P, dev(W))
    try:
        Y = torch.empty((N, M), dtype=torch.bfloat16, device="cuda")
        esp.espace_linear_forward(p, dev(X), Y)
        torch.cuda.synchronize()
        Yd = oracle.dense(f64(X), f64(W))
        err = np.linalg.norm(f64(Y) - Yd) / np.linalg.norm(Yd)
        assert err < 2e-2
    finally:
        esp.espace_proj_destroy(p)


def test_linear_forward_repeated_calls_and_scratch_growth(esp):
    K, M, L = 512, 512, 256
    P = synth.random_projection(K, L, seed=5)
    W = synth.weights(M, K, seed=5)
    p = esp.espace_proj_from_host(P, dev(W))
    model = synth.ActivationModel(K, seed=5)
    Pb = oracle.bf16_round(P)
    Wf_o = oracle.fold(Pb, f64(W))
    try:
        for N in (16, 300, 64, 700, 1):
            X = model.sample(N, chunk=N)
            Y = torch.empty((N, M), dtype=torch.bfloat16, device="cuda")
            esp.espace_linear_forward(p, dev(X), Y)
            torch.cuda.synchronize()
            Y_o, _, _ = oracle.forward(f64(X), Pb, f64(W), Wf=Wf_o)
            assert_y_close(Y, Y_o)
    finally:
        esp.espace_proj_destroy(p)


def test_single_token_forward_repeated_and_interleaved(esp):
    """Successive single tokens, and calls with more tokens in between, each match the
    oracle (the decode kernel's grid barrier and scratch are left ready for the next call);
    the same token twice agrees to within one bf16 ulp (partial sums meet in arrival order)."""
    K, M, L = 4096, 4096, 1024
    P = synth.random_projection(K, L, seed=8)
    W = synth.weights(M, K, seed=8)
    p = esp.espace_proj_from_host(P, dev(W))
    model = synth.ActivationModel(K, seed=8)
    Pb = oracle.bf16_round(P)
    Wf_o = oracle.fold(Pb, f64(W))
    try:
        X = model.sample(12, chunk=12)
        first = None
        for N, rows in ((1, slice(0, 1)), (1, slice(1, 2)), (8, slice(2, 10)), (1, slice(0, 1)), (1, slice(10, 11))):
            Xs = X[rows].contiguous()
            Y = torch.empty((N, M), dtype=torch.bfloat16, device="cuda")
            esp.espace_linear_forward(p, dev(Xs), Y)
            torch.cuda.synchronize()
            esp.espace_check()
            Y_o, _, _ = oracle.forward(f64(Xs), Pb, f64(W), Wf=Wf_o)
            assert_y_close(Y, Y_o)
            if rows == slice(0, 1):
                if first is None:
                    first = Y.clone()
                else:
                    ulp = (first.float() - Y.float()).abs() <= first.float().abs() * 2.0 ** -7
                    assert bool(ulp.all())
    finally:
        esp.espace_proj_destroy(p)


# ------------------------------------------------------------------ training view (Sec. 2.2)

def assert_close_normwise(A_gpu, A_ref, rel=Y_REL, mx_rel=Y_MAX):
    A = f64(A_gpu) if A_gpu.dtype == torch.bfloat16 else A_gpu.double().cpu().numpy()
    err = np.linalg.norm(A - A_ref) / max(np.linalg.norm(A_ref), 1e-300)
    mx = np.abs(A - A_ref).max() / max(np.abs(A_ref).max(), 1e-300)
    assert np.all(np.isfinite(A))
    assert err <= rel, f"normwise error {err:.3e}"
    assert mx <= mx_rel, f"max error {mx:.3e}"


TRAIN_CASES = [
    # (N, K, M, L)
    (300, 512, 776, 256),      # two launches forward, ragged M
    (1000, 1024, 1000, 512),   # fused forward, ragged N and M
    (129, 520, 264, 100),      # ragged K and L (Z padded to 128 columns)
    (2048, 1024, 2048, 512),   # several tiles each way
]


@pytest.mark.parametrize("N,K,M,L", TRAIN_CASES)
def test_train_forward_backward_matches_oracle(esp, N, K, M, L):
    """Y = W^T (P P^T X) with P static: the forward keeps Z, the backward returns dX (through
    P P^T) and dW = (dY^T Z) P^T, each against the oracle; then a weight update refolds W'."""
    seed = 4000 + N + K
    _, X, W = make_layer(K, M, N, seed=seed)
    P = synth.random_projection(K, L, seed=seed)
    r = np.random.default_rng(seed)
    dY = torch.from_numpy(r.standard_normal((N, M)).astype(np.float32)).to(torch.bfloat16)
    Lp = (L + 63) // 64 * 64
    p = esp.espace_proj_from_host(P, dev(W))
    try:
        Z = torch.full((N, Lp), float("nan"), dtype=torch.bfloat16, device="cuda")
        Y = torch.empty((N, M), dtype=torch.bfloat16, device="cuda")
        esp.espace_train_forward(p, dev(X), Z, Y)
        dX = torch.full((N, K), float("nan"), dtype=torch.bfloat16, device="cuda")
        dW = torch.full((M, K), float("nan"), dtype=torch.float32, device="cuda")
        esp.espace_train_backward(p, dev(dY), Z, dX)
        esp.espace_train_weight_grad(p, dW)
        torch.cuda.synchronize()
        esp.espace_check()
        Pb = oracle.bf16_round(P)
        Wf = oracle.fold(Pb, f64(W))
        Y_o, Z_o, _ = oracle.forward(f64(X), Pb, f64(W), Wf=Wf)
        Zg = f64(Z)
        assert np.all(Zg[:, L:] == 0)
        assert_close_normwise(Z[:, :L], Z_o)
        assert_y_close(Y, Y_o)
        # the backward products are checked from the oracle's own Z (the GPU's Z may differ
        # from it by isolated one-ulp roundings, within the tolerances)
        dX_o, dW_o = oracle.train_backward(f64(dY), Z_o, Pb, Wf)
        assert_close_normwise(dX, dX_o)
        assert_close_normwise(dW, dW_o)
        # two micro-batches of one step: the weight gradient sums over both (their tokens)
        X2 = make_layer(K, M, N, seed=seed + 2)[1]
        dY2 = torch.from_numpy(r.standard_normal((N, M)).astype(np.float32)).to(torch.bfloat16)
        Z2 = torch.empty_like(Z)
        esp.espace_train_forward(p, dev(X2), Z2, Y)
        esp.espace_train_backward(p, dev(dY), Z, dX)
        esp.espace_train_backward(p, dev(dY2), Z2, dX)
        esp.espace_train_weight_grad(p, dW)
        torch.cuda.synchronize()
        Z2_o = oracle.forward(f64(X2), Pb, f64(W), Wf=Wf)[1]
        both = np.concatenate([Z_o, Z2_o])
        _, dW_o2 = oracle.train_backward(np.concatenate([f64(dY), f64(dY2)]), both, Pb, Wf)
        assert_close_normwise(dW, dW_o2)
        # an optimizer step: new weights, W' refolded on the device
        W2 = synth.weights(M, K, seed=seed + 1)
        esp.espace_proj_refold(p, dev(W2))
        esp.espace_train_forward(p, dev(X), Z, Y)
        torch.cuda.synchronize()
        assert_y_close(Y, oracle.forward(f64(X), Pb, f64(W2))[0])
    finally:
        esp.espace_proj_destroy(p)


@pytest.mark.parametrize("N,K,M", [(300, 512, 776), (2048, 1024, 2048), (129, 136, 392)])
def test_dense_backward_matches_oracle(esp, N, K, M):
    _, X, W = make_layer(K, M, N, seed=5000 + N)
    r = np.random.default_rng(N)
    dY = torch.from_numpy(r.standard_normal((N, M)).astype(np.float32)).to(torch.bfloat16)
    dX = torch.empty((N, K), dtype=torch.bfloat16, device="cuda")
    dW = torch.empty((M, K), dtype=torch.float32, device="cuda")
    esp.espace_dense_backward(dev(dY), dev(X), dev(W), dX, dW)
    torch.cuda.synchronize()
    esp.espace_check()
    dX_o, dW_o = oracle.dense_backward(f64(dY), f64(X), f64(W))
    assert_close_normwise(dX, dX_o)
    assert_close_normwise(dW, dW_o, rel=1e-5, mx_rel=1e-4)
    esp.espace_dense_backward(dev(dY), dev(X), dev(W), dX, dW, accumulate=True)
    torch.cuda.synchronize()
    assert_close_normwise(dW, 2 * dW_o, rel=1e-5, mx_rel=1e-4)


# ------------------------------------------------------------------ NL-MSE calibration (Thm. 2)

def _unit_rows_bf16(A):
    A = f64(A)
    n = np.linalg.norm(A, axis=1, keepdims=True)
    return oracle.bf16_round(np.where(n > 0, A / np.where(n > 0, n, 1.0), 0.0))


@pytest.mark.parametrize("K,T", [(1040, 2048), (64, 300)])
def test_calib_nl_mse_split_reduction(esp, K, T):
    """NL-MSE terms against the oracle: at K = 1040 the SYRKs split their token reduction
    (2048 tokens, 15 upper tiles of a ragged K per problem, both problems in one launch) and
    the K x K products end in a ragged k-block padded with zero rows; at K = 64 the 1-CTA
    kernels run each product as its own launch."""
    Xs = synth.ActivationModel(K, seed=71).sample(T, stream="calib_tokens")
    Gs = (synth.ActivationModel(K, seed=72, outliers=0, lognormal_sigma=0.0)
          .sample(T, stream="calib_tokens", chunk=1) * 0.01).to(torch.bfloat16)
    h = esp.espace_calib_create(K)
    try:
        esp.espace_calib_accumulate_nl(h, dev(Xs), dev(Gs))
        C, n = esp.espace_calib_read(h, K)
        assert n == 1
    finally:
        esp.espace_calib_destroy(h)
    C_o = oracle.nl_mse_term(f64(Xs), f64(Gs))
    err = np.linalg.norm(C - C_o) / np.linalg.norm(C_o)
    assert err <= 1e-4, err


@pytest.mark.parametrize("normalized", [False, True])
def test_calib_nl_mse_matches_oracle(esp, normalized):
    """Three calibration sequences of activations and synthetic loss gradients: C (the mean
    of the per-sequence NL-MSE matrices) against the oracle, then the projection (ordered
    by |eigenvalue| when C is indefinite) and the forward with the library's P."""
    K, M, L, T, nseq, N = 512, 512, 128, 256, 3, 96
    xm = synth.ActivationModel(K, seed=61, outliers=5, lognormal_sigma=0.5)
    gm = synth.ActivationModel(K, seed=62, outliers=0, lognormal_sigma=0.0)
    Xs = [xm.sample(T, stream="calib_tokens", chunk=i) for i in range(nseq)]
    Gs = [gm.sample(T, stream="calib_tokens", chunk=i) * 0.01 for i in range(nseq)]
    Gs = [g.to(torch.bfloat16) for g in Gs]
    X = xm.sample(N)
    W = synth.weights(M, K, seed=61)
    h = esp.espace_calib_create(K)
    p = None
    try:
        for Xi, Gi in zip(Xs, Gs):
            esp.espace_calib_accumulate_nl(h, dev(Xi), dev(Gi), normalized)
        C, n = esp.espace_calib_read(h, K)
        assert n == nseq
        if normalized:
            # the library rounds the unit-norm rows to bf16 before the tensor-core products
            terms = [oracle.nl_mse_term(_unit_rows_bf16(Xi), _unit_rows_bf16(Gi)) for Xi, Gi in zip(Xs, Gs)]
        else:
            terms = [oracle.nl_mse_term(f64(Xi), f64(Gi)) for Xi, Gi in zip(Xs, Gs)]
        C_o = sum(terms) / nseq
        err = np.linalg.norm(C - C_o) / np.linalg.norm(C_o)
        assert err <= 1e-4, err
        with pytest.raises(esp.EspaceError):
            esp.espace_calib_accumulate(h, dev(Xs[0]))          # kinds do not mix
        p = esp.espace_build_projection(h, dev(W), L)
        w = esp.espace_proj_eigenvalues(p)
        w_o, V_o, _ = oracle.eigh(C_o)
        w_o, V_o = oracle.order_eigenpairs(w_o, V_o)
        scale = np.abs(w_o).max()
        if w_o[-1] < 0:
            assert np.all(np.diff(np.abs(w)) <= 1e-12 * scale)
        assert np.allclose(np.sort(w), np.sort(w_o), rtol=0, atol=2e-4 * scale)
        P_o = oracle.normalize_signs(V_o[:, :L])
        Pb = synth.bf16_to_f64(torch.from_numpy(esp.espace_proj_read_P(p).view(np.int16)).view(torch.bfloat16))
        gap = abs(w_o[L - 1]) - abs(w_o[L])
        proj = np.linalg.norm(Pb @ Pb.T - P_o @ P_o.T, 2)
        assert proj <= 2e-4 * np.linalg.norm(C_o) / gap + 2e-2, (proj, gap)
        Y = torch.empty((N, M), dtype=torch.bfloat16, device="cuda")
        esp.espace_linear_forward(p, dev(X), Y)
        torch.cuda.synchronize()
        esp.espace_check()
        assert_y_close(Y, oracle.forward(f64(X), Pb, f64(W))[0])
    finally:
        if p:
            esp.espace_proj_destroy(p)
        esp.espace_calib_destroy(h)


# ------------------------------------------------------------------ tensor-parallel ranks (App. B.2)

TP_CASES = [
    # (kind, tp, N, K, M, L)
    ("row", 4, 300, 1024, 776, 128),      # K / tp = 256, ragged M
    ("row", 3, 129, 576, 392, 64),        # three ranks (K / tp = 192), ragged N
    ("row", 8, 1000, 2048, 1000, 128),    # eight ranks, several row blocks
    ("row", 4, 1, 1024, 512, 64),         # one token
    ("column", 4, 300, 512, 1056, 128),   # M / tp = 264: rank blocks straddle 256-wide tiles
    ("column", 2, 257, 520, 784, 256),    # K not a multiple of 64, M / tp = 392
    ("column", 8, 64, 1024, 2048, 64),    # few tokens, eight ranks
]


@pytest.mark.parametrize("kind,tp,N,K,M,L", TP_CASES)
def test_tp_forward_matches_oracle(esp, kind, tp, N, K, M, L):
    """Each rank with its own projection: the folded layer (a dense product and a
    block-diagonal one) against the oracle's per-rank definition."""
    seed = 3000 + tp + N + K
    _, X, W = make_layer(K, M, N, seed=seed)
    r = np.random.default_rng(seed)
    Kr = K // tp if kind == "row" else K
    P = np.stack([synth.haar_orthonormal(r, Kr, L) for _ in range(tp)])
    code = esp.TP_ROW if kind == "row" else esp.TP_COLUMN
    p = esp.espace_proj_tp_from_host(code, P, dev(W))
    try:
        assert esp.espace_proj_tp_info(p) == (code, tp)
        assert esp.espace_linear_forward_launches(p, N) == 2
        Y = torch.full((N, M), float("nan"), dtype=torch.bfloat16, device="cuda")
        esp.espace_linear_forward(p, dev(X), Y)
        torch.cuda.synchronize()
        esp.espace_check()
        Pb = oracle.bf16_round(P)
        bits = esp.espace_proj_read_P(p)
        assert np.array_equal(synth.bf16_to_f64(torch.from_numpy(bits.view(np.int16)).view(torch.bfloat16)), Pb)
        Y_o = oracle.forward_tp(f64(X), Pb, f64(W), kind)
        assert_y_close(Y, Y_o)
    finally:
        esp.espace_proj_destroy(p)


def test_tp_identity_projections_reproduce_the_dense_layer(esp):
    """Row-parallel ranks with identity projections (L = K / tp): the folded layer is Eq. 1."""
    N, K, M, tp = 200, 512, 520, 4
    _, X, W = make_layer(K, M, N, seed=41)
    P = np.stack([np.eye(K // tp)] * tp)
    p = esp.espace_proj_tp_from_host(esp.TP_ROW, P, dev(W))
    try:
        Y = torch.empty((N, M), dtype=torch.bfloat16, device="cuda")
        esp.espace_linear_forward(p, dev(X), Y)
        Yd = torch.empty_like(Y)
        esp.espace_dense_forward(dev(X), dev(W), Yd)
        torch.cuda.synchronize()
        assert_y_close(Y, oracle.dense(f64(X), f64(W)))
        assert_y_close(Y, f64(Yd))
    finally:
        esp.espace_proj_destroy(p)


def test_build_projection_tp(esp):
    """Thm. 1 per rank from one calibration: row-parallel ranks solve C's diagonal blocks
    (eigenvalues and subspaces against the oracle, then the forward with the library's
    projections); column-parallel ranks all see C, so the handle is the plain layer."""
    K, M, L, tp, n, N = 1024, 776, 128, 4, 8192, 300
    Kr = K // tp
    model = synth.ActivationModel(K, seed=51, outliers=10, lognormal_sigma=0.5)
    Xc = model.sample(n, stream="calib_tokens")
    X = model.sample(N)
    W = synth.weights(M, K, seed=51)
    h = esp.espace_calib_create(K)
    p = q = None
    try:
        esp.espace_calib_accumulate(h, dev(Xc))
        p = esp.espace_build_projection_tp(h, dev(W), L, esp.TP_ROW, tp)
        assert esp.espace_proj_tp_info(p) == (esp.TP_ROW, tp)
        w = esp.espace_proj_eigenvalues(p).reshape(tp, Kr)
        S_o = oracle.autocorr_sum(f64(Xc))
        P_o, _, w_o = oracle.build_projection_tp(S_o, n, L, "row", tp)
        Pb = synth.bf16_to_f64(torch.from_numpy(esp.espace_proj_read_P(p).view(np.int16)).view(torch.bfloat16))
        for r in range(tp):
            assert np.all(np.diff(w[r]) <= 0)
            assert np.allclose(w[r], w_o[r], rtol=0, atol=1e-5 * w_o[r][0])
            gap = w_o[r][L - 1] - w_o[r][L]
            dC = 1e-5 * np.linalg.norm(S_o / n)
            proj = np.linalg.norm(Pb[r] @ Pb[r].T - P_o[r] @ P_o[r].T, 2)
            assert proj <= dC / gap + 2e-2, (r, proj, dC / gap)
        Y = torch.empty((N, M), dtype=torch.bfloat16, device="cuda")
        esp.espace_linear_forward(p, dev(X), Y)
        torch.cuda.synchronize()
        esp.espace_check()
        assert_y_close(Y, oracle.forward_tp(f64(X), Pb, f64(W), "row"))
        q = esp.espace_build_projection_tp(h, dev(W), L, esp.TP_COLUMN, tp)
        assert esp.espace_proj_tp_info(q) == (0, 1)
        assert esp.espace_proj_shape(q) == (K, M, L)
    finally:
        for handle in (p, q):
            if handle:
                esp.espace_proj_destroy(handle)
        esp.espace_calib_destroy(h)


@pytest.mark.slow
def test_llama2_qkv_prefill_full_size_sampled(esp):
    """K=4096, M=12288, L=2048, N=4096 (the Llama2 QKV prefill launch): all 12,288 outputs
    of 66 sampled tokens (the first, the last and 64 seeded ones) against the oracle."""
    K, M, L, N = 4096, 12288, 2048, 4096
    seed = synth.config_seed("llama2_qkv_prefill")
    model, X, W = make_layer(K, M, N, seed=seed)
    P = synth.random_projection(K, L, seed=seed)
    p = esp.espace_proj_from_host(P, dev(W))
    try:
        Y = torch.empty((N, M), dtype=torch.bfloat16, device="cuda")
        esp.espace_linear_forward(p, dev(X), Y)
        torch.cuda.synchronize()
        esp.espace_check()
        r = np.random.default_rng(seed)
        toks = np.unique(np.concatenate([[0, N - 1], r.choice(N, 64, replace=False)]))
        Pb = oracle.bf16_round(P)
        Wf_o = oracle.fold_matmul(Pb, f64(W))
        Z_o = oracle.project(f64(X[toks]), Pb)
        Y_o = oracle.contract(Z_o, Wf_o)
        assert_y_close(f64(Y[toks]), Y_o)
    finally:
        esp.espace_proj_destroy(p)


# ------------------------------------------------------------------------------ calibration (Eq. 4)

@pytest.mark.parametrize("K,n,chunks", [(512, 2048, 1), (136, 1000, 3), (1024, 4096, 2), (64, 7, 1)])
def test_calib_accumulate_matches_oracle(esp, K, n, chunks):
    model = synth.ActivationModel(K, seed=K + n, outliers=None if K >= 100 else 1)
    X = model.sample(n, stream="calib_tokens")
    h = esp.espace_calib_create(K)
    try:
        Xd = dev(X)
        bounds = np.linspace(0, n, chunks + 1).astype(int)
        for a, b in zip(bounds[:-1], bounds[1:]):
            esp.espace_calib_accumulate(h, Xd[a:b].contiguous())
        C, cnt = esp.espace_calib_read(h, K)
        esp.espace_check()
        assert cnt == n
        C_o = oracle.autocorr_sum(f64(X)) / n
        err = np.linalg.norm(C - C_o) / np.linalg.norm(C_o)
        assert err <= C_REL, f"C normwise error {err:.3e}"
        assert np.array_equal(C, C.T)
    finally:
        esp.espace_calib_destroy(h)


def test_calib_normalized_matches_oracle(esp):
    K, n = 256, 1500
    X = synth.ActivationModel(K, seed=9).sample(n, stream="calib_tokens")
    h = esp.espace_calib_create(K)
    try:
        esp.espace_calib_accumulate_normalized(h, dev(X))
        C, cnt = esp.espace_calib_read(h, K)
        # the library rounds the unit-norm tokens to bf16 before the tensor-core product
        Xf = f64(X)
        U = oracle.bf16_round(Xf / np.linalg.norm(Xf, axis=1, keepdims=True))
        C_o = oracle.autocorr_sum(U) / n
        err = np.linalg.norm(C - C_o) / np.linalg.norm(C_o)
        assert err <= 1e-4, err
        assert abs(np.trace(C) - 1.0) < 1e-2
    finally:
        esp.espace_calib_destroy(h)


def test_calib_export_import_and_shard_sum(esp):
    K = 128
    model = synth.ActivationModel(K, seed=3)
    X1, X2 = model.sample(700, chunk=1), model.sample(500, chunk=2)
    hs = [esp.espace_calib_create(K) for _ in range(3)]
    try:
        esp.espace_calib_accumulate(hs[0], dev(X1))
        esp.espace_calib_accumulate(hs[1], dev(X2))
        S1, n1 = esp.espace_calib_export(hs[0], K)
        S2, n2 = esp.espace_calib_export(hs[1], K)
        esp.espace_calib_import(hs[2], S1 + S2, n1 + n2)
        C, n = esp.espace_calib_read(hs[2], K)
        C_o = oracle.autocorr_sum(np.concatenate([f64(X1), f64(X2)])) / 1200
        assert n == 1200
        assert np.linalg.norm(C - C_o) / np.linalg.norm(C_o) <= C_REL
        esp.espace_calib_reset(hs[0])
        S0, n0 = esp.espace_calib_export(hs[0], K)
        assert n0 == 0 and not np.any(np.triu(S0))
        with pytest.raises(esp.EspaceError) as e:      # C = S / n is undefined for n = 0
            esp.espace_calib_read(hs[0], K)
        assert e.value.code == 6
    finally:
        for h in hs:
            esp.espace_calib_destroy(h)


# ------------------------------------------------------------------------------ build (Thm. 1)

def test_build_projection_tiny_config(esp):
    cfg = synth.CONFIGS["tiny"]
    K, M, L, N, n = cfg["K"], cfg["M"], cfg["L"], cfg["N"], cfg["calib_tokens"]
    seed = synth.config_seed("tiny")
    model = synth.ActivationModel(K, seed=seed, outliers=cfg["outliers"], lognormal_sigma=cfg["lognormal_sigma"])
    Xc = model.sample(n, stream="calib_tokens")
    X = model.sample(N)
    W = synth.weights(M, K, seed=seed)
    h = esp.espace_calib_create(K)
    p = None
    try:
        esp.espace_calib_accumulate(h, dev(Xc))
        p = esp.espace_build_projection(h, dev(W), L)
        w = esp.espace_proj_eigenvalues(p)
        S_o = oracle.autocorr_sum(f64(Xc))
        P_o, Pb_o, w_o, _ = oracle.build_projection(S_o, n, L)
        assert np.all(np.diff(w) <= 0)
        assert np.allclose(w, w_o, rtol=0, atol=1e-5 * w_o[0])
        Pb = synth.bf16_to_f64(torch.from_numpy(esp.espace_proj_read_P(p).view(np.int16)).view(torch.bfloat16))
        # same subspace: projector distance within Davis-Kahan (C error / gap) plus bf16 rounding
        gap = w_o[L - 1] - w_o[L]
        dC = 1e-5 * np.linalg.norm(S_o / n)
        proj = np.linalg.norm(Pb @ Pb.T - P_o @ P_o.T, 2)
        assert proj <= dC / gap + 2e-2, (proj, dC / gap)
        # Theorem 1 on the calibration tokens with the library's (bf16) P
        mse = oracle.projection_mse(f64(Xc), Pb)
        assert mse <= np.sum(w_o[L:]) * 1.05 + 1e-3 * np.sum(w_o)
        # end to end: forward with the library's projection against the oracle fed that P
        Y = torch.empty((N, M), dtype=torch.bfloat16, device="cuda")
        esp.espace_linear_forward(p, dev(X), Y)
        torch.cuda.synchronize()
        Y_o, _, _ = oracle.forward(f64(X), Pb, f64(W))
        assert_y_close(Y, Y_o)
        esp.espace_check()
    finally:
        if p:
            esp.espace_proj_destroy(p)
        esp.espace_calib_destroy(h)


@pytest.mark.parametrize("normalized", [False, True])
def test_build_projection_go_tiny_config(esp, normalized):
    """Thm. 2 (GO-MSE, and with Cor. 1's normalized calibration its L2-normalized variant):
    eigenvalues of C = C_X C_W + C_W C_X and the L-dimensional subspace against the oracle,
    then the forward with the library's P."""
    cfg = synth.CONFIGS["tiny"]
    K, M, L, N, n = cfg["K"], cfg["M"], cfg["L"], cfg["N"], cfg["calib_tokens"]
    seed = synth.config_seed("tiny")
    model = synth.ActivationModel(K, seed=seed, outliers=cfg["outliers"], lognormal_sigma=cfg["lognormal_sigma"])
    Xc = model.sample(n, stream="calib_tokens")
    X = model.sample(N)
    W = synth.weights(M, K, seed=seed)
    h = esp.espace_calib_create(K)
    p = None
    try:
        if normalized:
            # the library rounds the unit-norm tokens to bf16 before the tensor-core product
            # (its norms in fp32: an occasional rounding differs, hence the looser tolerance)
            esp.espace_calib_accumulate_normalized(h, dev(Xc))
            Xf = f64(Xc)
            S_o = oracle.autocorr_sum(oracle.bf16_round(Xf / np.linalg.norm(Xf, axis=1, keepdims=True)))
            tol = 1e-4
        else:
            esp.espace_calib_accumulate(h, dev(Xc))
            S_o = oracle.autocorr_sum(f64(Xc))
            tol = 1e-5
        p = esp.espace_build_projection_go(h, dev(W), L)
        w = esp.espace_proj_eigenvalues(p)
        P_o, Pb_o, w_o, _ = oracle.build_projection_go(S_o, n, f64(W), L)
        scale = np.abs(w_o).max()
        assert np.all(np.diff(np.abs(w)) <= 1e-12 * scale)          # ordered by magnitude
        assert np.allclose(np.sort(w), np.sort(w_o), rtol=0, atol=tol * scale)
        Pb = synth.bf16_to_f64(torch.from_numpy(esp.espace_proj_read_P(p).view(np.int16)).view(torch.bfloat16))
        # same subspace: projector distance within Davis-Kahan (C error / gap at the cut) plus
        # the bf16 rounding of P
        gap = abs(w_o[L - 1]) - abs(w_o[L])
        C_o = oracle.go_mse_matrix(S_o / n, f64(W))
        dC = tol * np.linalg.norm(C_o)
        proj = np.linalg.norm(Pb @ Pb.T - P_o @ P_o.T, 2)
        assert proj <= dC / gap + 2e-2, (proj, dC / gap)
        Y = torch.empty((N, M), dtype=torch.bfloat16, device="cuda")
        esp.espace_linear_forward(p, dev(X), Y)
        torch.cuda.synchronize()
        Y_o, _, _ = oracle.forward(f64(X), Pb, f64(W))
        assert_y_close(Y, Y_o)
        esp.espace_check()
    finally:
        if p:
            esp.espace_proj_destroy(p)
        esp.espace_calib_destroy(h)


def test_proj_export_import_roundtrip(esp):
    K, M, L = 256, 128, 96
    P = synth.random_projection(K, L, seed=21)
    W = synth.weights(M, K, seed=21)
    p = esp.espace_proj_from_host(P, dev(W))
    q = None
    try:
        PT, WfT, ev = esp.espace_proj_export(p)
        q = esp.espace_proj_import(K, M, L, PT, WfT, ev)
        X = synth.ActivationModel(K, seed=21).sample(33)
        Y1 = torch.empty((33, M), dtype=torch.bfloat16, device="cuda")
        Y2 = torch.empty_like(Y1)
        esp.espace_linear_forward(p, dev(X), Y1)
        esp.espace_linear_forward(q, dev(X), Y2)
        torch.cuda.synchronize()
        assert torch.equal(Y1, Y2)
    finally:
        esp.espace_proj_destroy(p)
        if q:
            esp.espace_proj_destroy(q)


# ------------------------------------------------------------------------------ errors

def test_argument_errors_launch_nothing(esp):
    K, M, L = 128, 64, 32
    P = synth.random_projection(K, L, seed=1)
    W = dev(synth.weights(M, K, seed=1))
    p = esp.espace_proj_from_host(P, W)
    try:
        X = torch.zeros((4, K), dtype=torch.bfloat16, device="cuda")
        Y = torch.zeros((4, M), dtype=torch.bfloat16, device="cuda")
        # misaligned pointer
        buf = torch.zeros(4 * K + 8, dtype=torch.bfloat16, device="cuda")
        rc = esp.lib.espace_linear_forward(p, buf.data_ptr() + 2, 4, Y.data_ptr(), None)
        assert rc == 3
        # small-N path refused beyond its limits
        Xb = torch.zeros((64, K), dtype=torch.bfloat16, device="cuda")
        Yb = torch.zeros((64, M), dtype=torch.bfloat16, device="cuda")
        with pytest.raises(esp.EspaceError) as e:
            esp.espace_linear_forward_path(p, Xb, Yb, esp.PATH_SMALL_N)
        assert e.value.code == 2
        # N = 0 is a no-op
        assert esp.lib.espace_linear_forward(p, X.data_ptr(), 0, Y.data_ptr(), None) == 0
        with pytest.raises(esp.EspaceError):
            esp.espace_proj_from_host(np.zeros((K, K + 1)), W)
        with pytest.raises(esp.EspaceError) as e:
            esp.espace_dense_forward(torch.zeros((4, 12), dtype=torch.bfloat16, device="cuda"),
                                     torch.zeros((8, 12), dtype=torch.bfloat16, device="cuda"),
                                     torch.zeros((4, 8), dtype=torch.bfloat16, device="cuda"))
        assert e.value.code == 2
        esp.espace_check()
    finally:
        esp.espace_proj_destroy(p)


def test_empty_batches_are_no_ops(esp):
    """Zero tokens (an empty tensor, whose data pointer is null) is accepted by every entry
    point that takes a batch and changes nothing; the dense backward without accumulation
    still clears dW."""
    K, M, L = 128, 64, 32
    W = dev(synth.weights(M, K, seed=2))
    p = esp.espace_proj_from_host(synth.random_projection(K, L, seed=2), W)
    h = esp.espace_calib_create(K)
    try:
        bf = dict(dtype=torch.bfloat16, device="cuda")
        X0, Y0 = torch.empty((0, K), **bf), torch.empty((0, M), **bf)
        Z0 = torch.empty((0, 64), **bf)
        esp.espace_linear_forward(p, X0, Y0)
        esp.espace_linear_forward_host(p, X0.cpu(), Y0.cpu())
        esp.espace_dense_forward(X0, W, Y0)
        esp.espace_train_forward(p, X0, Z0, Y0)
        esp.espace_train_backward(p, Y0, Z0, X0)
        esp.espace_calib_accumulate(h, X0)
        S, n = esp.espace_calib_export(h, K)
        assert n == 0 and not np.any(S)
        with pytest.raises(esp.EspaceError) as e:
            esp.espace_calib_read(h, K)                  # C = S / n needs tokens
        assert e.value.code == 6
        dW = torch.full((M, K), 7.0, dtype=torch.float32, device="cuda")
        esp.espace_dense_backward(Y0, X0, W, X0, dW, accumulate=True)
        torch.cuda.synchronize()
        assert bool((dW == 7.0).all())
        esp.espace_dense_backward(Y0, X0, W, X0, dW, accumulate=False)
        torch.cuda.synchronize()
        assert not bool(dW.any())
        esp.espace_check()
    finally:
        esp.espace_calib_destroy(h)
        esp.espace_proj_destroy(p)


def test_bounded_wait_reports_timeout_and_context_survives(esp):
    esp.espace_check()
    esp.espace_debug_wait_timeout(2_000_000)          # 2 ms
    with pytest.raises(esp.EspaceError) as e:
        esp.espace_check()
    assert e.value.code == 5
    esp.espace_check()                                 # cleared
    # the context is still usable
    X = torch.ones((8, 64), dtype=torch.bfloat16, device="cuda")
    W = torch.ones((16, 64), dtype=torch.bfloat16, device="cuda")
    Y = torch.empty((8, 16), dtype=torch.bfloat16, device="cuda")
    esp.espace_dense_forward(X, W, Y)
    torch.cuda.synchronize()
    assert torch.all(Y.float() == 64.0)


def _layer_and_reference(esp, K, M, L, N, seed):
    _, X, W = make_layer(K, M, N, seed=seed)
    P = synth.random_projection(K, L, seed=seed)
    p = esp.espace_proj_from_host(P, dev(W))
    Y_o = oracle.forward(f64(X), oracle.bf16_round(P), f64(W))[0]
    return p, dev(X), Y_o


def test_fused_forward_completes_while_other_work_holds_half_the_sms(esp):
    """The fused forward's CTA pairs draw their work items from a ticket, Z tiles first: a
    pair that draws a Y tile waits only for Z tiles already drawn by running pairs. So with
    half of the SMs held by another stream's kernel (300 ms), the forward runs on the other
    half within a 50 ms wait limit and gives the right result; with the items split among
    the pairs in advance, a resident pair would wait for Z tiles of a pair that cannot
    start, until the limit."""
    K, M, L, N = 1024, 2048, 512, 2048
    p, Xd, Y_o = _layer_and_reference(esp, K, M, L, N, seed=77)
    try:
        assert esp.espace_linear_forward_launches(p, N) == 1
        Y = torch.empty((N, M), dtype=torch.bfloat16, device="cuda")
        esp.espace_linear_forward(p, Xd, Y)            # scratch allocated here
        torch.cuda.synchronize()
        esp.espace_check()
        Y.fill_(float("nan"))
        sms = torch.cuda.get_device_properties(0).multi_processor_count
        side = torch.cuda.Stream()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        torch.cuda.synchronize()
        esp.espace_set_wait_limit_ns(50_000_000)
        try:
            esp.espace_debug_occupy(sms // 2, 300_000_000, side)
            time.sleep(0.02)                            # the holding CTAs are resident
            a.record()
            esp.espace_linear_forward(p, Xd, Y)
            b.record()
            torch.cuda.synchronize()
        finally:
            esp.espace_set_wait_limit_ns(4_000_000_000)
        esp.espace_check()                              # no wait gave up
        assert a.elapsed_time(b) < 150.0                # it ran beside the holding kernel
        assert_y_close(Y, Y_o)
    finally:
        esp.espace_proj_destroy(p)


@pytest.mark.parametrize("N", [64, 200])
def test_few_token_forward_completes_while_other_work_holds_half_the_sms(esp, N):
    """The few-token products are launches whose CTAs never wait for one another (each item's
    tile, or split partial, is the CTA's own; the partials are added by the next launch). With
    half of the SMs held by another stream's kernel (300 ms) they run on the other half
    within a 50 ms wait limit and give the right result, for the projected layer and for the
    dense one."""
    K, M, L = 2048, 2048, 1024
    p, Xd, Y_o = _layer_and_reference(esp, K, M, L, N, seed=81)
    try:
        Y = torch.empty((N, M), dtype=torch.bfloat16, device="cuda")
        esp.espace_linear_forward(p, Xd, Y)            # workspace allocated here
        W = dev(synth.weights(M, K, seed=81))
        Yd = torch.empty((N, M), dtype=torch.bfloat16, device="cuda")
        esp.espace_dense_forward(Xd, W, Yd)
        torch.cuda.synchronize()
        esp.espace_check()
        Y.fill_(float("nan"))
        Yd.fill_(float("nan"))
        sms = torch.cuda.get_device_properties(0).multi_processor_count
        side = torch.cuda.Stream()
        torch.cuda.synchronize()
        esp.espace_set_wait_limit_ns(50_000_000)
        try:
            esp.espace_debug_occupy(sms // 2, 300_000_000, side)
            time.sleep(0.02)                            # the holding CTAs are resident
            esp.espace_linear_forward(p, Xd, Y)
            esp.espace_dense_forward(Xd, W, Yd)
            torch.cuda.synchronize()
        finally:
            esp.espace_set_wait_limit_ns(4_000_000_000)
        esp.espace_check()                              # no wait gave up
        assert_y_close(Y, Y_o)
        assert_y_close(Yd, oracle.dense(f64(Xd.cpu()), f64(W.cpu())))
    finally:
        esp.espace_proj_destroy(p)


@pytest.mark.parametrize("N", [1, 8, 24])
def test_decode_forward_completes_while_other_work_holds_half_the_sms(esp, N):
    """The decode kernel's two products meet at a grid barrier, so it is a cooperative
    launch: with half of the SMs held by another stream's kernel (300 ms), it starts once all
    of its CTAs can be resident, and none of its bounded waits counts the time before that.
    Within a 50 ms wait limit it completes with the right result, and so does the next call
    on the handle (24 tokens: the decode kernel forced, two token tiles)."""
    K, M, L = 2048, 2048, 1024
    p, Xd, Y_o = _layer_and_reference(esp, K, M, L, N, seed=79)
    try:
        path = esp.PATH_SMALL_N if N > 16 else esp.PATH_AUTO
        assert esp.espace_linear_forward_launches(p, N, path) == 1
        Y = torch.empty((N, M), dtype=torch.bfloat16, device="cuda")
        esp.espace_linear_forward_path(p, Xd, Y, path)
        torch.cuda.synchronize()
        esp.espace_check()
        assert_y_close(Y, Y_o)
        Y.fill_(float("nan"))
        sms = torch.cuda.get_device_properties(0).multi_processor_count
        side = torch.cuda.Stream()
        torch.cuda.synchronize()
        esp.espace_set_wait_limit_ns(50_000_000)
        try:
            esp.espace_debug_occupy(sms // 2, 300_000_000, side)
            time.sleep(0.02)                            # the holding CTAs are resident
            esp.espace_linear_forward_path(p, Xd, Y, path)
            torch.cuda.synchronize()
        finally:
            esp.espace_set_wait_limit_ns(4_000_000_000)
        esp.espace_check()                              # no wait gave up
        assert_y_close(Y, Y_o)
        Y.fill_(float("nan"))
        esp.espace_linear_forward_path(p, Xd, Y, path)  # and the next call on the handle
        torch.cuda.synchronize()
        esp.espace_check()
        assert_y_close(Y, Y_o)
    finally:
        esp.espace_proj_destroy(p)


@pytest.mark.parametrize("N,K,L", [(2048, 1024, 512), (4, 1024, 512), (4, 2048, 1536), (64, 1024, 512),
                                   (200, 2048, 1024)])
def test_forward_after_a_launch_that_gave_up(esp, N, K, L):
    """A launch whose waits give up (a 2 us limit) leaves the handle's counters consistent:
    the fused kernel's last CTA zeroes its readiness counters, ticket and exit counter on
    every exit path, every CTA of the decode kernel arrives once at its grid barrier (whose
    second phase runs over one k-block of Z at L = 512, two at L = 1536), and the few-token
    products (64 and 200 tokens: swapped launches with split reductions) keep no state
    between launches. The timeout is reported, and the next forwards on the same handle are
    right."""
    M = 2048
    p, Xd, Y_o = _layer_and_reference(esp, K, M, L, N, seed=78)
    try:
        Y = torch.empty((N, M), dtype=torch.bfloat16, device="cuda")
        esp.espace_linear_forward(p, Xd, Y)
        torch.cuda.synchronize()
        esp.espace_check()
        assert_y_close(Y, Y_o)
        esp.espace_set_wait_limit_ns(2_000)
        try:
            esp.espace_linear_forward(p, Xd, Y)
            torch.cuda.synchronize()
        finally:
            esp.espace_set_wait_limit_ns(4_000_000_000)
        if N > 256:
            with pytest.raises(esp.EspaceError) as e:
                esp.espace_check()
            assert e.value.code == 5
        else:
            try:
                esp.espace_check()
            except esp.EspaceError as e:                # a short launch may finish in time
                assert e.code == 5
        for _ in range(2):
            Y.fill_(float("nan"))
            esp.espace_linear_forward(p, Xd, Y)
            torch.cuda.synchronize()
            esp.espace_check()
            assert_y_close(Y, Y_o)
    finally:
        esp.espace_proj_destroy(p)


# ------------------------------------------------------------------------------ degenerate calibrations

def test_build_projection_rank_deficient_calibration(esp):
    """Fewer calibration tokens (64) than features (256): C has rank 64, so with L = 128 the
    projection keeps all of the calibration variance (Thm. 1: the discarded eigenvalues are
    zero) and its extra columns span part of C's null space, where any orthonormal choice is
    right. Checked: eigenvalues against the oracle (zero beyond the rank, within the fp32
    sums), orthonormal P within bf16 rounding, the MSE of Eq. 6 on the calibration tokens
    near zero, and the forward with the library's P."""
    K, M, L, n, N = 256, 192, 128, 64, 100
    model = synth.ActivationModel(K, seed=31)
    Xc = model.sample(n, stream="calib_tokens")
    X = model.sample(N)
    W = synth.weights(M, K, seed=31)
    h = esp.espace_calib_create(K)
    p = None
    try:
        esp.espace_calib_accumulate(h, dev(Xc))
        p = esp.espace_build_projection(h, dev(W), L)
        w = esp.espace_proj_eigenvalues(p)
        Pb = synth.bf16_to_f64(torch.from_numpy(esp.espace_proj_read_P(p).view(np.int16)).view(torch.bfloat16))
        Y = torch.empty((N, M), dtype=torch.bfloat16, device="cuda")
        esp.espace_linear_forward(p, dev(X), Y)
        torch.cuda.synchronize()
        esp.espace_check()
    finally:
        if p:
            esp.espace_proj_destroy(p)
        esp.espace_calib_destroy(h)
    w_o = oracle.eigh(oracle.autocorr_sum(f64(Xc)) / n)[0]
    assert np.allclose(w, w_o, rtol=0, atol=1e-5 * w_o[0])
    assert np.all(np.abs(w[n:]) <= 1e-5 * w_o[0])
    assert np.abs(Pb.T @ Pb - np.eye(L)).max() < 2e-2
    mse = oracle.projection_mse(f64(Xc), Pb)
    total = oracle.projection_mse(f64(Xc), np.zeros((K, 1)))          # E ||x||^2
    assert mse <= 1e-4 * total, (mse, total)
    assert_y_close(Y, oracle.forward(f64(X), Pb, f64(W))[0])


def test_build_projection_from_all_zero_calibration(esp):
    """All-zero calibration tokens: C = 0, every eigenvalue is zero and every orthonormal P
    is optimal (Thm. 1). The build must still give orthonormal columns (bf16) and a working
    layer: the forward matches the oracle fed the library's P."""
    K, M, L, n, N = 64, 96, 16, 100, 40
    h = esp.espace_calib_create(K)
    p = None
    try:
        esp.espace_calib_accumulate(h, torch.zeros((n, K), dtype=torch.bfloat16, device="cuda"))
        p = esp.espace_build_projection(h, dev(synth.weights(M, K, seed=32)), L)
        w = esp.espace_proj_eigenvalues(p)
        Pb = synth.bf16_to_f64(torch.from_numpy(esp.espace_proj_read_P(p).view(np.int16)).view(torch.bfloat16))
        X = synth.ActivationModel(K, seed=32).sample(N)
        Y = torch.empty((N, M), dtype=torch.bfloat16, device="cuda")
        esp.espace_linear_forward(p, dev(X), Y)
        torch.cuda.synchronize()
        esp.espace_check()
    finally:
        if p:
            esp.espace_proj_destroy(p)
        esp.espace_calib_destroy(h)
    assert np.all(w == 0)
    assert np.abs(Pb.T @ Pb - np.eye(L)).max() < 2e-2
    assert_y_close(Y, oracle.forward(f64(X), Pb, f64(synth.weights(M, K, seed=32)))[0])


@pytest.mark.parametrize("N", [4, 24, 64, 200])
def test_few_token_chain_reads_each_input_after_it_is_written(esp, N):
    """A chain of few-token layers on one stream with no synchronization between them: each
    layer's input is the previous one's output (buffers filled with NaN first), projected and
    dense layers interleaved. The few-token launches may start while the previous kernel
    finishes and load their weights early, but must read their tokens only after it has
    completed: every output must equal the oracle applied to the input it was given."""
    K = M = 1024
    L = 512
    torch.cuda.synchronize()
    Ws = [synth.weights(M, K, seed=90 + i) for i in range(4)]
    ps = [esp.espace_proj_from_host(synth.random_projection(K, L, seed=90 + i), dev(Ws[i])) for i in range(3)]
    try:
        X0 = dev(synth.ActivationModel(K, seed=90).sample(N))
        W3 = dev(Ws[3])
        outs = [torch.full((N, M), float("nan"), dtype=torch.bfloat16, device="cuda") for _ in range(6)]
        torch.cuda.synchronize()
        x = X0
        kinds = []
        for i, y in enumerate(outs):
            if i % 2 == 1:
                esp.espace_dense_forward(x, W3, y)
                kinds.append("dense")
            else:
                esp.espace_linear_forward(ps[i // 2], x, y)
                kinds.append(i // 2)
            x = y
        torch.cuda.synchronize()
        esp.espace_check()
        x = X0
        for kind, y in zip(kinds, outs):
            xf = f64(x)
            if kind == "dense":
                ref = oracle.dense(xf, f64(Ws[3]))
            else:
                Pb = oracle.bf16_round(synth.random_projection(K, L, seed=90 + kind))
                ref = oracle.forward(xf, Pb, f64(Ws[kind]))[0]
            assert_y_close(y, ref)
            x = y
    finally:
        for p in ps:
            esp.espace_proj_destroy(p)
