"""Pins of the oracle's byte accounting (Sec. 3.4, Eq. 5) and record layout:
the paper's worked Qwen2.5-3B sidecar example, hand-computed record sizes for
every workload, and one record's bytes derived by hand from the layout."""
import json
import os

import numpy as np
import pytest

GOLD = os.path.join(os.path.dirname(__file__), "golden")


def test_paper_sidecar_example(orc):
    g = json.load(open(os.path.join(GOLD, "paper_sidecar_example.json")))
    n_scope = g["layers"] * sum(r * c for r, c in g["module_shapes"])
    assert n_scope == 2_434_793_472
    T = n_scope // g["C"]
    # a 7-byte record holds ceil(log2 T) + ceil(log2 S) + b_e + P*b bits for every
    # exponent width 1 <= b_e <= 8, including ours (8)
    for b_e in range(1, 9):
        prm = orc.params(C=g["C"], P=g["P"], b=g["b"], S=g["S"], b_e=b_e)
        assert orc.record_bytes(prm, T) == g["record_bytes"]
    prm = orc.params(C=g["C"], P=g["P"], b=g["b"], S=g["S"], b_e=9)
    assert orc.record_bytes(prm, T) == 8
    assert orc.header_bytes(g["n_modules"]) == g["header_bytes"]
    side = g["header_bytes"] + g["K"] * g["record_bytes"]
    assert side == g["sidecar_bytes"]
    assert round(8 * side / n_scope, 3) == g["added_scope_bpw_printed"]
    # that stream fits the 0.162 bits/weight budget of Eq. 5 (floor(r N / 8) bytes)
    assert orc.budget_bytes(0.162, n_scope) >= side


@pytest.mark.parametrize("T,S,b_e,expect", [
    (2048, 256, 8, 6),            # small single matrix, power-of-two scale: 11+8+8+16 = 43 bits
    (2048, 256, 16, 7),           # same with a binary16 scale: 51 bits
    (1_204_224, 4096, 8, 8),      # one Qwen2.5-3B layer: 21+12+8+16 = 57 bits
    (43_352_064, 4096, 8, 8),     # 36 layers: 26+12+8+16 = 62 bits
    (101_957_632, 4096, 8, 8),    # Qwen2.5-7B stack: 27+12+8+16 = 63 bits
    (487_587_840, 4096, 8, 9),    # Qwen2.5-32B stack: 29+12+8+16 = 65 bits
    (1, 1, 8, 3),                 # degenerate: no tile or seed bits, 8+16 = 24 bits
])
def test_record_sizes(orc, T, S, b_e, expect):
    prm = orc.params(C=64, P=4, b=4, S=S, b_e=b_e, scale_mode=1 if b_e == 16 else 0)
    assert orc.record_bytes(prm, T) == expect


def test_record_bytes_by_hand(orc):
    """tile 5, seed 3, e = -13, codes (-1, -6, -5, 6) with T = 2048, S = 256, b_e = 8:
    bits LSB-first: tile 10100000000 | seed 11000000 | e 11001111 | 1111 0101 1101 0110."""
    prm = orc.params(C=64, P=4, b=4, S=256, b_e=8)
    cand = np.zeros(1, orc.CANDIDATE_DTYPE)[0]
    cand["gain"] = 1.0
    cand["seed"] = 3
    cand["scale"] = -13
    cand["code"][:4] = [-1, -6, -5, 6]
    rec = orc.pack_record(prm, 2048, 5, cand)
    assert rec == bytes([0x05, 0x18, 0x98, 0x7F, 0x5D, 0x03])
    tile, back = orc.unpack_record(prm, 2048, rec)
    assert tile == 5 and back["seed"] == 3 and back["scale"] == -13
    assert list(back["code"][:4]) == [-1, -6, -5, 6]
    # the same record with e_bias = -20: the field holds e - e_bias = 7 (11100000)
    prm = orc.params(C=64, P=4, b=4, S=256, b_e=8, e_bias=-20)
    rec = orc.pack_record(prm, 2048, 5, cand)
    assert rec == bytes([0x05, 0x18, 0x38, 0x78, 0x5D, 0x03])
    tile, back = orc.unpack_record(prm, 2048, rec)
    assert tile == 5 and back["scale"] == -13


def test_record_round_trip_extremes(orc):
    rng = np.random.default_rng(0)
    for C, P, b, S, b_e, e_bias, smode in [(64, 4, 4, 4096, 8, 0, 0), (16, 8, 8, 65536, 3, -12, 0),
                                          (128, 2, 2, 2, 16, 0, 1), (8, 1, 5, 1, 1, -10, 0)]:
        prm = orc.params(C=C, P=P, b=b, S=S, b_e=b_e, e_bias=e_bias, scale_mode=smode)
        T = int(rng.integers(1, 10**9))
        qmax = 2 ** (b - 1) - 1
        lo = max(e_bias - 2 ** (b_e - 1), -126)
        hi = min(e_bias + 2 ** (b_e - 1) - 1, 126)
        for _ in range(200):
            c = np.zeros(1, orc.CANDIDATE_DTYPE)[0]
            c["seed"] = rng.integers(0, S)
            c["scale"] = rng.integers(0, 0x7c00) if smode else rng.integers(lo, hi + 1)
            c["code"][:P] = rng.integers(-qmax, qmax + 1, P)
            tile = int(rng.integers(0, T))
            rec = orc.pack_record(prm, T, tile, c)
            assert len(rec) == orc.record_bytes(prm, T)
            t2, c2 = orc.unpack_record(prm, T, rec)
            assert t2 == tile and c2["seed"] == c["seed"] and c2["scale"] == c["scale"]
            assert np.array_equal(c2["code"], c["code"])
