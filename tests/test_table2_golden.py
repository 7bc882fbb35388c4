"""Table 2's printed configurations (App. B.2) against the paper's compression metric and
its rule for choosing L, and the per-layer configurations the Table 2 benchmark uses.

The compression rate (Sec. 4.1) counts, for a projected layer, the entries of P and of
W' = P^T W instead of those of W. A column-parallel layer's ranks see the same inputs and
share one P (K x L) while W' spans all N outputs; a row-parallel layer's ranks each hold
their own P_r (K/tp x L) and W'_r (L x N). The paper's N (outputs) is this library's M.
"""
from __future__ import annotations

import os

import pytest

import synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "table2_configurations.txt")

# Rows where the printed values disagree with each other, and the reading taken.
#  - llama2_13b fc2: the printed L = 1024 gives 20.7 % per rank (K/tp = 1728, N = 5120),
#    against the printed 60 % and the rule of App. B.2 (at least 50 % per layer); L = 512
#    gives 60.4 %. Read as L = 512.
#  - nemotron4_15b proj: printed 67 %, but its shape and L are those of gpt3_22b proj,
#    printed 63 % (62.5 % computed). The printed L is kept.
#  - llama2_7b fc1: printed 69 %, computed 70.35 %. The printed L is kept.
L_READING = {("llama2_13b", "fc2"): 512}


def _rows():
    rows = []
    with open(GOLDEN) as f:
        for line in f:
            line = line.strip()
            if not line or line.startswith("#"):
                continue
            model, tp, layer, kind, K, N, L, pct = line.split()
            rows.append(dict(model=model, tp=int(tp), layer=layer, kind=kind, K=int(K), N=int(N), L=int(L),
                             pct=float(pct)))
    return rows


def compression(kind: str, tp: int, K: int, N: int, L: int) -> float:
    """Percentage of a layer's weight entries removed by ESPACE (Sec. 4.1's count)."""
    if kind == "column":
        return 100.0 * (1.0 - L * (K + N) / (K * N))
    k = K // tp
    return 100.0 * (1.0 - L * (k + N) / (k * N))


def test_fixture_holds_all_six_models_and_four_layers():
    rows = _rows()
    assert len(rows) == 24
    assert sorted({r["model"] for r in rows}) == sorted(synth.TABLE2)
    for r in rows:
        assert r["kind"] == ("column" if r["layer"] in ("qkv", "fc1") else "row")
        assert r["K"] % r["tp"] == 0 and r["N"] % r["tp"] == 0


def test_worked_example_square_layer_at_quarter_rank_is_half_compressed():
    """Sec. 2.2: with N = K and L = K/4, ESPACE stores half of the entries."""
    for K in (1024, 4096, 6144):
        assert compression("column", 1, K, K, K // 4) == pytest.approx(50.0, abs=1e-12)


def test_printed_compression_follows_from_the_printed_shapes():
    by_key = {(r["model"], r["layer"]): r for r in _rows()}
    for key, r in by_key.items():
        c = compression(r["kind"], r["tp"], r["K"], r["N"], r["L"])
        if key == ("llama2_13b", "fc2"):
            assert c == pytest.approx(20.7, abs=0.05)               # far from the printed 60
            c512 = compression(r["kind"], r["tp"], r["K"], r["N"], L_READING[key])
            assert abs(c512 - r["pct"]) <= 1.0
        elif key == ("nemotron4_15b", "proj"):
            twin = by_key[("gpt3_22b", "proj")]
            assert (r["tp"], r["K"], r["N"], r["L"]) == (twin["tp"], twin["K"], twin["N"], twin["L"])
            assert c == pytest.approx(62.5, abs=1e-9)
            assert abs(c - twin["pct"]) <= 1.0 and abs(c - r["pct"]) > 4.0
        elif key == ("llama2_7b", "fc1"):
            assert abs(c - r["pct"]) <= 1.5
        else:
            assert abs(c - r["pct"]) <= 1.0, (key, c, r["pct"])


def test_rank_rule_of_appendix_b2():
    """L is a power of two and gives at least 50 % per layer, except the QKV layers of
    Llama2-13B and Nemotron4 (about 45 %, stated as the exception); the printed L of
    Llama2-13B's FC2 breaks the rule, its reading keeps it."""
    for r in _rows():
        key = (r["model"], r["layer"])
        L = L_READING.get(key, r["L"])
        assert L & (L - 1) == 0
        c = compression(r["kind"], r["tp"], r["K"], r["N"], L)
        if key in (("llama2_13b", "qkv"), ("nemotron4_15b", "qkv")):
            assert 40.0 <= c < 50.0
        else:
            assert c >= 50.0 - 1e-9, (key, c)
    r = next(r for r in _rows() if (r["model"], r["layer"]) == ("llama2_13b", "fc2"))
    assert compression(r["kind"], r["tp"], r["K"], r["N"], r["L"]) < 50.0


def test_benchmark_configurations_match_the_table():
    for r in _rows():
        cfg = synth.TABLE2[r["model"]]
        assert cfg["tp"] == r["tp"]
        layers = {name: (kind, K, M, L) for name, kind, K, M, L in cfg["layers"]}
        L = L_READING.get((r["model"], r["layer"]), r["L"])
        assert layers[r["layer"]] == (r["kind"], r["K"], r["N"], L)
