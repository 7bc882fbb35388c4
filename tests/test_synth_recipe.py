"""The synthetic input recipe that stands in for the paper's activations and weights: a
power-law spectrum i^-0.8, a seeded orthonormal rotation (Haar, or four Householder
reflectors with a signed permutation), log-normal channel scales, round(0.01 K) outlier
channels x20, W ~ N(0, 1/K), and the gated down-projection input silu(a) * b. Every draw
is seeded by (seed, stream, chunk)."""
from __future__ import annotations

import math

import numpy as np
import pytest
import torch

import synth


@pytest.mark.parametrize("rotation", ["haar", "householder"])
def test_rotation_is_orthonormal(rotation):
    K = 96
    m = synth.ActivationModel(K, seed=3, rotation=rotation)
    QT = m._rotate(np.eye(K, dtype=np.float32)).astype(np.float64)
    assert np.allclose(QT @ QT.T, np.eye(K), atol=1e-5)
    assert not np.allclose(QT, np.eye(K), atol=1e-2)                # it does rotate


def test_outlier_channels_count_and_gain():
    for K, want in ((64, 1), (512, 5), (4096, 41), (11008, 110)):
        m = synth.ActivationModel(K, seed=4, lognormal_sigma=0.0, rotation="householder")
        assert len(m.outlier_channels) == want
        scale = m.channel_scale
        assert np.all(scale[m.outlier_channels] == 20.0)
        mask = np.ones(K, dtype=bool)
        mask[m.outlier_channels] = False
        assert np.all(scale[mask] == 1.0)
    m = synth.ActivationModel(512, seed=4, outliers=0, lognormal_sigma=0.5)
    logs = np.log(m.channel_scale)
    assert abs(logs.mean()) < 0.1 and abs(logs.std() - 0.5) < 0.06


def test_draws_are_deterministic_per_stream_and_chunk():
    m = synth.ActivationModel(128, seed=5)
    a = m.sample(64, stream="calib_tokens", chunk=2)
    assert torch.equal(a, synth.ActivationModel(128, seed=5).sample(64, stream="calib_tokens", chunk=2))
    assert not torch.equal(a, m.sample(64, stream="calib_tokens", chunk=3))
    assert not torch.equal(a, m.sample(64, stream="eval_tokens", chunk=2))
    assert not torch.equal(a, synth.ActivationModel(128, seed=6).sample(64, stream="calib_tokens", chunk=2))
    assert a.dtype == torch.bfloat16 and a.shape == (64, 128)


def test_second_moment_converges_to_the_population_form():
    """E[x^T x] = diag(c) Q diag(s^2) Q^T diag(c) for rows x = (g * s) Q^T * c."""
    K, n = 24, 200_000
    m = synth.ActivationModel(K, seed=7, outliers=1, lognormal_sigma=0.5, rotation="householder")
    QT = m._rotate(np.eye(K, dtype=np.float32)).astype(np.float64)
    c = m.channel_scale
    C_pop = (QT.T * m.spectrum ** 2) @ QT
    C_pop = c[:, None] * C_pop * c[None, :]
    X = m.sample_f32(n).astype(np.float64)
    C = X.T @ X / n
    assert np.linalg.norm(C - C_pop) <= 0.02 * np.linalg.norm(C_pop)


def test_weights_and_gated_input():
    M, K = 256, 512
    W = synth.weights(M, K, seed=8).float().numpy()
    assert abs(W.mean()) < 5.0 * math.sqrt(1.0 / K) / math.sqrt(M * K)   # five standard errors
    assert abs(W.var() * K - 1.0) < 0.02
    m = synth.ActivationModel(64, seed=9)
    g = m.sample_gated(32, chunk=1).float().numpy()
    a = m.sample_f32(32, "gate_a", 1).astype(np.float64)
    b = m.sample_f32(32, "gate_b", 1).astype(np.float64)
    ref = a / (1.0 + np.exp(-a)) * b
    assert np.allclose(g, ref, rtol=2 ** -7, atol=1e-6 * np.abs(ref).max())
