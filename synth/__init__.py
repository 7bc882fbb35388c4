"""Seeded synthetic inputs shaped like the linear layers of GPT3, Llama2 and Nemotron4.

This module only draws random numbers and arranges them into bf16 tensors. It holds no step
of the projected-linear method (no autocorrelation, no eigen-solve, no projection, no fold):
the CUDA path and the fp64 oracle both consume what it produces, and neither shares any
other code with the other.

Recipe (the paper measures on Wikitext-103 / MTNLG activations of trained models, which are
not available; these inputs stand in for them with the same layer shapes):

* activations ``X[n, :] = ((g * s) @ Q^T) * c * o`` with ``g`` iid N(0, 1) per token,
  a power-law spectrum ``s_i = i^-decay`` (``decay = 0.8``), a seeded random orthonormal
  rotation ``Q`` (Haar: QR of a Gaussian matrix with the sign fix, for K <= 4096; above
  that a product of four seeded Householder reflectors composed with a seeded signed
  permutation, which is orthonormal and costs O(K) per token and reflector), log-normal
  per-channel scales ``c_k = exp(sigma * xi_k)`` and ``outliers`` channels scaled by
  ``outlier_gain``; the product is rounded to bf16 (round-to-nearest-even, by torch);
* weights ``W[m, :]`` iid N(0, 1/K), stored ``[M][K]`` (PyTorch ``nn.Linear`` layout);
* a gated input ``silu(a) * b`` for down-projections, with ``a`` and ``b`` drawn
  independently from the activation model and combined in fp32 before the bf16 cast;
* random orthonormal ``K x L`` matrices (QR of a Gaussian), used where a test needs some
  projection without running an eigen-solve.

Every stream is a numpy Philox generator keyed by ``(seed, stream id, chunk)``, so a
chunk of tokens is reproducible on its own and calibration and evaluation tokens are
independent draws.
"""
from __future__ import annotations

import math
from dataclasses import dataclass

import numpy as np
import torch

BASE_SEED = 0x24105437

_STREAMS = {
    "rotation": 1,
    "channel_scale": 2,
    "outliers": 3,
    "weights": 4,
    "calib_tokens": 5,
    "eval_tokens": 6,
    "projection": 7,
    "gate_a": 8,
    "gate_b": 9,
    "misc": 10,
}


def generator(seed: int, stream: str, chunk: int = 0) -> np.random.Generator:
    """Philox generator for one named stream (and chunk) of one seed."""
    return np.random.Generator(
        np.random.Philox(np.random.SeedSequence([int(seed), _STREAMS[stream], int(chunk)])))


def to_bf16(a: np.ndarray) -> torch.Tensor:
    """fp32/fp64 numpy array -> bf16 torch tensor (CPU), rounded to nearest even by torch."""
    return torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32)).to(torch.bfloat16)


def haar_orthonormal(rng: np.random.Generator, rows: int, cols: int) -> np.ndarray:
    """Random ``rows x cols`` matrix with orthonormal columns (QR of a Gaussian, sign fixed)."""
    g = rng.standard_normal((rows, cols))
    q, r = np.linalg.qr(g)
    d = np.sign(np.diag(r))
    d[d == 0] = 1.0
    return q * d


@dataclass
class ActivationModel:
    """Seeded generator of activation tokens ``x`` in ``R^K`` (see the module docstring)."""

    K: int
    seed: int = BASE_SEED
    decay: float = 0.8
    outliers: int | None = None      # None -> round(0.01 * K)
    outlier_gain: float = 20.0
    lognormal_sigma: float = 0.5     # 0 -> no per-channel scales
    rotation: str = "auto"           # "haar", "householder" or "auto" (haar for K <= 4096)

    def __post_init__(self):
        K = self.K
        self.spectrum = np.arange(1, K + 1, dtype=np.float64) ** (-self.decay)
        rot = self.rotation
        if rot == "auto":
            rot = "haar" if K <= 4096 else "householder"
        self._rot = rot
        rg = generator(self.seed, "rotation")
        if rot == "haar":
            self.Q = haar_orthonormal(rg, K, K)
            self._QT32 = np.ascontiguousarray(self.Q.T, dtype=np.float32)
        elif rot == "householder":
            self.Q = None
            v = rg.standard_normal((4, K))
            self._reflectors = (v / np.linalg.norm(v, axis=1, keepdims=True)).astype(np.float32)
            self._perm = rg.permutation(K)
            self._signs = np.where(rg.random(K) < 0.5, -1.0, 1.0).astype(np.float32)
        else:
            raise ValueError(f"unknown rotation {rot!r}")
        scale = np.ones(K)
        if self.lognormal_sigma > 0:
            scale = np.exp(self.lognormal_sigma * generator(self.seed, "channel_scale").standard_normal(K))
        n_out = int(round(0.01 * K)) if self.outliers is None else int(self.outliers)
        if n_out > 0:
            idx = generator(self.seed, "outliers").permutation(K)[:n_out]
            scale[idx] *= self.outlier_gain
            self.outlier_channels = np.sort(idx)
        else:
            self.outlier_channels = np.zeros(0, dtype=np.int64)
        self.channel_scale = scale

    def _rotate(self, y: np.ndarray) -> np.ndarray:
        """Rows of ``y`` times ``Q^T`` (y is float32 [n, K])."""
        if self._rot == "haar":
            return y @ self._QT32
        for v in self._reflectors:              # y <- y (I - 2 v v^T), four times
            y = y - 2.0 * np.outer(y @ v, v).astype(np.float32)
        return y[:, self._perm] * self._signs

    def sample_f32(self, n: int, stream: str = "eval_tokens", chunk: int = 0) -> np.ndarray:
        g = generator(self.seed, stream, chunk).standard_normal((n, self.K), dtype=np.float32)
        y = g * self.spectrum.astype(np.float32)
        return self._rotate(y) * self.channel_scale.astype(np.float32)

    def sample(self, n: int, stream: str = "eval_tokens", chunk: int = 0) -> torch.Tensor:
        """``n`` tokens as a bf16 ``[n, K]`` CPU tensor."""
        return to_bf16(self.sample_f32(n, stream, chunk))

    def sample_device(self, n: int, stream: str = "eval_tokens", chunk: int = 0,
                      device: str = "cuda") -> torch.Tensor:
        """Same recipe drawn on the GPU with torch's Philox generator (a different random
        stream from ``sample``): for benchmark inputs too large to draw on the host. Not
        used where an oracle value is compared."""
        gen = torch.Generator(device=device)
        gen.manual_seed((int(self.seed) * 1000003 + _STREAMS[stream] * 7919 + int(chunk)) % (1 << 63))
        g = torch.randn((n, self.K), generator=gen, device=device, dtype=torch.float32)
        y = g * torch.as_tensor(self.spectrum, dtype=torch.float32, device=device)
        if self._rot == "haar":
            if getattr(self, "_QT_dev", None) is None or self._QT_dev.device != y.device:
                self._QT_dev = torch.as_tensor(self._QT32, device=device)
            y = y @ self._QT_dev
        else:
            for v in self._reflectors:
                vt = torch.as_tensor(v, device=device)
                y = y - 2.0 * (y @ vt)[:, None] * vt[None, :]
            y = y[:, torch.as_tensor(self._perm, device=device)] * torch.as_tensor(self._signs, device=device)
        y = y * torch.as_tensor(self.channel_scale, dtype=torch.float32, device=device)
        return y.to(torch.bfloat16)

    def sample_gated(self, n: int, chunk: int = 0) -> torch.Tensor:
        """Down-projection input ``silu(a) * b`` (fp32, then bf16) with independent a, b."""
        a = self.sample_f32(n, "gate_a", chunk)
        b = self.sample_f32(n, "gate_b", chunk)
        silu = a / (1.0 + np.exp(-a))
        return to_bf16(silu * b)


def weights(M: int, K: int, seed: int = BASE_SEED, chunk: int = 0) -> torch.Tensor:
    """``W`` as bf16 ``[M, K]`` (PyTorch Linear layout), iid N(0, 1/K)."""
    w = generator(seed, "weights", chunk).standard_normal((M, K), dtype=np.float32)
    return to_bf16(w * np.float32(1.0 / math.sqrt(K)))


def weights_device(M: int, K: int, seed: int = BASE_SEED, chunk: int = 0,
                   device: str = "cuda") -> torch.Tensor:
    """``W`` drawn on the GPU (benchmark inputs only; see ``ActivationModel.sample_device``)."""
    gen = torch.Generator(device=device)
    gen.manual_seed((int(seed) * 1000003 + _STREAMS["weights"] * 7919 + int(chunk)) % (1 << 63))
    w = torch.randn((M, K), generator=gen, device=device, dtype=torch.float32)
    return (w * (1.0 / math.sqrt(K))).to(torch.bfloat16)


def structured_projection(K: int, L: int, seed: int = BASE_SEED) -> np.ndarray:
    """A seeded ``K x L`` fp64 matrix with orthonormal columns built in O(K L): the first L
    columns of (four Householder reflectors) x (signed permutation). Used at shapes where a
    Gaussian QR would take minutes."""
    rg = generator(seed, "projection", 1)
    perm = rg.permutation(K)[:L]
    signs = np.where(rg.random(L) < 0.5, -1.0, 1.0)
    Q = np.zeros((K, L))
    Q[perm, np.arange(L)] = signs
    for _ in range(4):
        v = rg.standard_normal(K)
        v /= np.linalg.norm(v)
        Q -= 2.0 * np.outer(v, v @ Q)
    return Q


def random_projection(K: int, L: int, seed: int = BASE_SEED) -> np.ndarray:
    """A seeded ``K x L`` fp64 matrix with orthonormal columns."""
    return haar_orthonormal(generator(seed, "projection"), K, L)


def bf16_bits(t: torch.Tensor) -> np.ndarray:
    """Raw uint16 bit patterns of a bf16 CPU tensor."""
    return t.contiguous().view(torch.int16).numpy().view(np.uint16)


def bf16_to_f64(t: torch.Tensor) -> np.ndarray:
    """Exact fp64 values of a bf16 tensor."""
    return t.to(torch.float64).numpy()


# The five workloads the benchmark and the parity tests use, in the order they are quoted.
CONFIGS = {
    "tiny": dict(K=512, M=512, L=256, N=128, calib_tokens=2048, outliers=4, lognormal_sigma=0.0),
    "llama2_qkv_prefill": dict(K=4096, M=12288, L=2048, N=4096, calib_tokens=65536),
    "llama2_mlp_gate_up": dict(K=4096, M=22016, L=2048, N=8192, calib_tokens=65536),
    "llama2_mlp_down": dict(K=11008, M=4096, L=5504, N=8192, calib_tokens=65536, gated=True),
    "gpt3_22b_qkv": dict(K=6144, M=18432, L=3072, N=16384, calib_tokens=1048576),
    "gpt3_22b_fc1": dict(K=6144, M=24576, L=3072, N=16384, calib_tokens=1048576),
    "gpt3_22b_fc2": dict(K=24576, M=6144, L=12288, N=16384, calib_tokens=1048576),
}

# Decode-shaped Llama2-7B stack at rank L = K/2, swept over token counts.
DECODE_LAYERS = {
    "qkv": (4096, 12288),
    "o": (4096, 4096),
    "gate_up": (4096, 22016),
    "down": (11008, 4096),
}
DECODE_TOKENS = (1, 8, 32, 128, 512)

# Per-layer ESPACE configurations of Table 2 (App. B.2): per model the tensor-parallel rank
# count, the sequence length of the GEMM latency measurement (App. B.4: batch 1, 2048
# tokens for GPT3, 4096 for Llama2 and Nemotron4), and per layer (name, kind, K, M, L)
# with K, M the whole layer's input and output widths and L the per-rank rank; QKV and
# FC1 are column-parallel, the attention projection and FC2 row-parallel. Also Table 1's
# total GEMM latency reduction of the most compressed variant, on A100. Llama2-13B's FC2
# is printed with L = 1024 but also with 60 % compression, which only L = 512 gives per
# rank (1024 gives 21 %, below the table's own 50 % rule); L = 512 is taken.
TABLE2 = {
    "gpt3_1.3b": dict(tp=1, seq=2048, paper_reduction=0.34, layers=[
        ("qkv", "column", 2048, 6144, 512), ("proj", "row", 2048, 2048, 512),
        ("fc1", "column", 2048, 8192, 512), ("fc2", "row", 8192, 2048, 512)]),
    "gpt3_8b": dict(tp=4, seq=2048, paper_reduction=0.44, layers=[
        ("qkv", "column", 4096, 12288, 1024), ("proj", "row", 4096, 4096, 256),
        ("fc1", "column", 4096, 16384, 1024), ("fc2", "row", 16384, 4096, 1024)]),
    "gpt3_22b": dict(tp=8, seq=2048, paper_reduction=0.49, layers=[
        ("qkv", "column", 6144, 18432, 2048), ("proj", "row", 6144, 6144, 256),
        ("fc1", "column", 6144, 24576, 2048), ("fc2", "row", 24576, 6144, 1024)]),
    "llama2_7b": dict(tp=4, seq=4096, paper_reduction=0.46, layers=[
        ("qkv", "column", 4096, 12288, 1024), ("proj", "row", 4096, 4096, 256),
        ("fc1", "column", 4096, 22016, 1024), ("fc2", "row", 11008, 4096, 512)]),
    "llama2_13b": dict(tp=8, seq=4096, paper_reduction=0.36, layers=[
        ("qkv", "column", 5120, 15360, 2048), ("proj", "row", 5120, 5120, 256),
        ("fc1", "column", 5120, 27648, 2048), ("fc2", "row", 13824, 5120, 512)]),
    "nemotron4_15b": dict(tp=8, seq=4096, paper_reduction=0.46, layers=[
        ("qkv", "column", 6144, 8192, 2048), ("proj", "row", 6144, 6144, 256),
        ("fc1", "column", 6144, 24576, 2048), ("fc2", "row", 24576, 6144, 1024)]),
}


def config_seed(name: str) -> int:
    return BASE_SEED + list(CONFIGS).index(name)
